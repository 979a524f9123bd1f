"""bench.py's work model (the algorithmic bytes and flops behind `roofline` and
`round_roofline`), checked against the tensors the synthetic generator makes and
against the figures quoted for the Qwen3-8B shape."""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2609_37029_gb300 import synth  # noqa: E402

PROJ = ["fuse"] + ["qkv", "o_proj", "gate_up", "down"]


def _weight_bytes_and_flops(s, w):
    """Projection weight bytes and 2 M N K flops read off the generated tensors."""
    es = w["lm_head"].element_size()
    M = s.C * s.B
    byts, flops = w["fuse"].numel() * es, 2.0 * s.C * w["fuse"].numel()
    for lw in w["layers"]:
        for k in ("wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down"):
            byts += lw[k].numel() * es
            flops += 2.0 * M * lw[k].numel()
    byts += w["lm_head"].numel() * es
    flops += 2.0 * M * w["lm_head"].numel()
    return byts, flops


def test_gemm_model_counts_every_generated_projection_weight_once():
    s = synth.SMALL
    w = synth.make_weights(s)
    es = 2
    names = ["fuse"] + ["qkv", "o_proj", "gate_up", "down"] * s.D + ["lm_head"]
    model_b = model_f = 0.0
    for n in names:
        b, f = bench.gemm_work(s, n)
        # strip the activation and output bytes: what is left is the weight stream
        N_K = {"fuse": (s.H, s.L * s.H), "qkv": ((s.nq + 2 * s.nkv) * s.d, s.H), "o_proj": (s.H, s.nq * s.d),
               "gate_up": (2 * s.F, s.H), "down": (s.H, s.F), "lm_head": (s.V, s.H)}[n]
        model_b += N_K[0] * N_K[1] * es
        model_f += f
    want_b, want_f = _weight_bytes_and_flops(s, w)
    assert model_b == want_b
    assert model_f == want_f


def test_lm_head_launch_bytes_at_qwen3_8b():
    s = synth.Q8B
    b, f = bench.gemm_work(s, "lm_head")
    # bf16 weights 151936 x 4096, bf16 activations 256 x 4096, fp32 logits 256 x 151936
    assert b == 151936 * 4096 * 2 + 256 * 4096 * 2 + 256 * 151936 * 4 == 1402339328
    assert f == 2.0 * 256 * 151936 * 4096


def test_round_model_grows_with_the_accepted_rows_only_through_the_view_update():
    s = synth.Q8B
    b1, f1 = bench.round_work(s, 1.0)
    b2, f2 = bench.round_work(s, 2.0)
    kv = s.nkv * s.d
    # one more accepted row per request: its K and V read, and written to the window ring
    assert b2 - b1 == s.C * s.L * 2 * kv * 2 * 2
    # and the R summary queries score it and take its value: 4 d flops per (query, row)
    assert f2 - f1 == 4.0 * s.C * s.L * s.nq * s.R * s.d
    gemm_bytes = sum(bench.gemm_work(s, n)[0] for n in ["fuse"] + PROJ[1:] * s.D + ["lm_head"])
    assert 3.6e9 < gemm_bytes < b1 < 4.0e9          # the GEMMs' 3.69 GB dominate the round
