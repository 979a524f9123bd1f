"""Block-diffusion drafter forward (oracle side, fp64).  Test infrastructure only.

Restates Sec. 2.3 ("Proposal Model") and App. A.1 ("Drafter Forward Pass"):

1. boundary state: c_t = W_fuse [h^{l_1}; ...; h^{l_L}] -- a learned projection
   fusing the tapped-layer hidden states at the decoding boundary (Sec. 2.2).
2. input slots: slot 0 encodes the committed token a, slots 1..B-1 a mask
   embedding; each is combined with a within-block positional encoding and c_t
   (Sec. 2.3).  Reading: the three are added.
3. D Qwen3-style layers (App. B.1).  Draft layer j reads tapped layer l(j).  At
   each layer the block attends, with one softmax, over
   K = [K^b; K^w; G], V = [V^b; V^w; M_t] (Eq. draft-context), bidirectionally
   inside the block.
4. frozen target final norm and vocabulary head give the base logits z^(0) of
   all B slots in parallel (Sec. 2.3, Eq. block-diffusion).

Readings where the paper is silent (each listed in the design notes):
* layer pairing l(j) = floor(j * L / D) (identity when D = |L|, Sec. 2.3);
* Qwen3 block: RMSNorm (eps) -> q, k, v projections -> per-head RMSNorm of q and
  k -> rotary embedding (rotate-half form, base theta) of block q and k at
  absolute positions t + i (0-based; the committed token a sits at position t)
  -> attention -> output projection + residual -> RMSNorm -> SwiGLU MLP +
  residual; no biases;
* window keys arrive from the target already rotated; summary keys G are used
  raw, and no norm is applied to window or summary keys.
"""
from __future__ import annotations

import numpy as np


def _f64(a):
    return np.asarray(a, dtype=np.float64)


class OracleWeights:
    """fp64 copies of the drafter weights (numpy inputs, [out][in] linear layout)."""

    def __init__(self, w: dict):
        self._embed = w["embed"]                      # gathered row by row
        self.final_norm = _f64(w["final_norm"])
        self.lm_head = _f64(w["lm_head"])
        self.fuse = _f64(w["fuse"])
        self.pos = _f64(w["pos"])
        self.mask_emb = _f64(w["mask_emb"])
        self.G = _f64(w["G"])
        self.Ec = _f64(w["Ec"])
        self.Wc = _f64(w["Wc"])
        self.layers = [{k: _f64(v) for k, v in lw.items()} for lw in w["layers"]]

    def embed_row(self, tok):
        return _f64(self._embed[tok])


def rmsnorm(x, w, eps):
    """x / sqrt(mean(x^2) + eps) * w over the last axis (Qwen3 RMSNorm)."""
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * w


def silu(x):
    return x / (1.0 + np.exp(-x))


def rope(x, pos, theta):
    """Rotary embedding, rotate-half pairing (i, i + d/2), frequency theta^(-2i/d).

    x: [B][heads][d]; pos: [B] absolute positions.
    """
    d = x.shape[-1]
    half = d // 2
    inv_freq = theta ** (-(2.0 * np.arange(half, dtype=np.float64)) / d)
    ang = np.asarray(pos, dtype=np.float64)[:, None] * inv_freq[None, :]
    cos = np.cos(ang)[:, None, :]
    sin = np.sin(ang)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * cos - x2 * sin, x2 * cos + x1 * sin], axis=-1)


def context_attention(q, kb, vb, kw, vw, Gl, ml, d):
    """Eq. draft-context: each block query attends over [K^b; K^w; G] with values [V^b; V^w; M].

    q: [B][nq][d]; kb, vb: [B][nkv][d]; kw, vw: [n_w][nkv][d] (window, any order);
    Gl, ml: [nq][R][d] (summary keys and values of this layer).  One softmax
    (scale 1/sqrt(d)) across all three sources; no mask inside the block.
    """
    B, nq, _ = q.shape
    rep = nq // kb.shape[1]
    out = np.empty_like(q)
    for h in range(nq):
        g = h // rep
        K = np.concatenate([kb[:, g], kw[:, g], Gl[h]], axis=0)
        V = np.concatenate([vb[:, g], vw[:, g], ml[h]], axis=0)
        s = q[:, h] @ K.T / np.sqrt(d)
        s = s - s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p /= p.sum(axis=1, keepdims=True)
        out[:, h] = p @ V
    return out


def boundary_state(cfg, w: OracleWeights, hb_b):
    """c_t = W_fuse [h^{l_1}; ...; h^{l_L}] (Sec. 2.2), hb_b: [L][H]."""
    return w.fuse @ hb_b.reshape(-1)


def draft_layer(cfg, lw, x, pos, kw, vw, Gl, ml):
    """One Qwen3-style draft layer over the B block rows x [B][H]."""
    B = x.shape[0]
    eps = cfg.rms_eps
    xn = rmsnorm(x, lw["in_norm"], eps)
    q = (xn @ lw["wq"].T).reshape(B, cfg.nq, cfg.d)
    k = (xn @ lw["wk"].T).reshape(B, cfg.nkv, cfg.d)
    v = (xn @ lw["wv"].T).reshape(B, cfg.nkv, cfg.d)
    q = rope(rmsnorm(q, lw["q_norm"], eps), pos, cfg.rope_theta)
    k = rope(rmsnorm(k, lw["k_norm"], eps), pos, cfg.rope_theta)
    o = context_attention(q, k, v, kw, vw, Gl, ml, cfg.d)
    x = x + o.reshape(B, cfg.nq * cfg.d) @ lw["wo"].T
    xn = rmsnorm(x, lw["post_norm"], eps)
    x = x + (silu(xn @ lw["w_gate"].T) * (xn @ lw["w_up"].T)) @ lw["w_down"].T
    return x


def draft_hidden(cfg, st, w: OracleWeights, block_tokens, b):
    """Final hidden rows [B][H] of request b (before the frozen final norm).

    The "w/o boundary state" variant of the ablation (Sec. 3.4, Fig. 5) drops
    c_t from the input slots: x_i = E[u_i] + P_i.  (W = 0 and R = 0 are the
    variants without the recent window and without the global summary.)
    """
    emb = np.stack([w.embed_row(int(u)) if int(u) >= 0 else w.mask_emb
                    for u in block_tokens[b]])
    x = emb + w.pos
    if not getattr(cfg, "no_boundary", False):
        x = x + boundary_state(cfg, w, st.hb[b])[None, :]
    pos = int(st.t[b]) + np.arange(cfg.B)
    for j in range(cfg.D):
        l = cfg.layer_map[j]
        x = draft_layer(cfg, w.layers[j], x, pos, st.win_k[b][l], st.win_v[b][l],
                        w.G[l], st.m[b, l])
    return x


def draft_base_logits(cfg, st, w: OracleWeights, block_tokens, reqs=None):
    """Base logits z^(0) [len(reqs)][B][V] of the requested rows (all requests by default)."""
    reqs = range(cfg.C) if reqs is None else reqs
    out = []
    for b in reqs:
        x = draft_hidden(cfg, st, w, block_tokens, b)
        out.append(rmsnorm(x, w.final_norm, cfg.rms_eps) @ w.lm_head.T)
    return np.stack(out)
