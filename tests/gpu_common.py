"""Shared helpers of the GPU parity tests (CUDA path through the C ABI vs the oracle)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_37029_gb300 import synth


def lsp_lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2609_37029_gb300 import build
    build.build()
    from paper_2609_37029_gb300 import lsp
    return lsp


def f64(t):
    return t.detach().to("cpu", torch.float64).numpy()


def np_weights(w):
    """numpy (exact fp32 upcast) copies of a synth weight dict for the oracle."""
    conv = lambda t: t.detach().float().cpu().numpy()
    out = {k: conv(v) for k, v in w.items() if k != "layers"}
    out["layers"] = [{k: conv(v) for k, v in lw.items()} for lw in w["layers"]]
    return out


def cuda_weights(w):
    out = {k: v.cuda() for k, v in w.items() if k != "layers"}
    out["layers"] = [{k: v.cuda() for k, v in lw.items()} for lw in w["layers"]]
    return out


def export_state(lsp, st, s):
    """Interface arrays of a state, in the documented export layout."""
    cfg = lsp.make_config(s)
    n = lsp.lsp_state_bytes(cfg)
    buf = torch.empty(n, dtype=torch.uint8)
    lsp.lsp_state_export(st, buf)
    dt = s.torch_dtype
    es = 2 if s.dtype == "bf16" else 4
    sizes = [("win_k", s.C * s.L * s.nkv * s.W * s.d * es, dt, (s.C, s.L, s.nkv, s.W, s.d)),
             ("win_v", s.C * s.L * s.nkv * s.W * s.d * es, dt, (s.C, s.L, s.nkv, s.W, s.d)),
             ("m", s.C * s.L * s.nq * s.R * s.d * 4, torch.float32, (s.C, s.L, s.nq, s.R, s.d)),
             ("eta", s.C * s.L * s.nq * s.R * 4, torch.float32, (s.C, s.L, s.nq, s.R)),
             ("h", 0 if s.no_boundary else s.C * s.L * s.H * es, dt, (s.C, s.L, 0 if s.no_boundary else s.H)),
             ("t", s.C * 8, torch.int64, (s.C,))]
    out, off = {}, 0
    for name, nb, t, shp in sizes:
        out[name] = buf[off:off + nb].view(t).view(shp).clone()
        off += nb
    assert off == n
    return out


def window_in_prefix_order(ring, t, W):
    """Ring slots -> rows oldest-first (prefix row p lives in slot p mod W)."""
    cnt = min(t, W)
    return np.stack([ring[..., p % W, :] for p in range(t - cnt, t)], axis=-2) if cnt else ring[..., :0, :]


def fold_chunk(lsp, st, ost, s, G_np, k, v, h, acc):
    """Apply one view update to the GPU state and the oracle state."""
    lsp.lsp_view_update(st, k.cuda(), v.cuda(), h.cuda(), acc.cuda())
    oracle.view_update(s, ost, G_np, f64(k), f64(v), f64(h), acc.numpy())


def check_view_state(lsp, st, ost, s, atol_m=1e-4):
    ex = export_state(lsp, st, s)
    assert list(ex["t"].numpy()) == list(ost.t)
    np.testing.assert_allclose(ex["m"].double().numpy(), ost.m, rtol=0, atol=atol_m)
    np.testing.assert_allclose(ex["eta"].double().numpy(), ost.eta, rtol=0, atol=atol_m * 10)
    if not s.no_boundary:                                      # the variant keeps no boundary
        assert np.array_equal(f64(ex["h"]), ost.hb)
    wk, wv = f64(ex["win_k"]), f64(ex["win_v"])
    for b in range(s.C):
        t = int(ost.t[b])
        for l in range(s.L):
            gk = window_in_prefix_order(wk[b, l], t, s.W)       # [nkv][n][d]
            gv = window_in_prefix_order(wv[b, l], t, s.W)
            assert np.array_equal(gk.transpose(1, 0, 2), ost.win_k[b][l])
            assert np.array_equal(gv.transpose(1, 0, 2), ost.win_v[b][l])
    return ex
