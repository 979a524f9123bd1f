"""Workload shapes and seeded synthetic inputs for the drafting round.

This module holds sizes and random-number recipes only: no step of the drafting
computation (view extraction, drafter forward, sampling) is written here, so the
CUDA path and the fp64 oracle can both draw their inputs from it without sharing
any of the method's arithmetic.

Recipes (all seeded, all synthetic; the paper's LongSpec / CodeSpan / LongSWE
prefixes and its trained weights are not available, so these stand in for them):

* weights: every projection, embedding, positional table, mask embedding and the
  low-rank correction factors E_c, W_c are N(0, 0.02); the summary queries G are
  N(0, 1/d) as in the paper's initialisation (App. B.2, "Summary queries"); RMSNorm
  weights are 1 + N(0, 0.1) so that a swapped norm weight is visible in tests.
* target features (K rows, V rows, boundary hidden h) are i.i.d. N(0, 1); the
  "small" shape multiplies each tapped layer by an RMS scale drawn U[0.5, 2]; the
  "large" shape multiplies a fixed 1% subset of channel indices by 20.
* accepted lengths per request and round are U[1, delta_max]; the committed token
  `a` of each request is U[0, V).
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass, field

import torch


@dataclass(frozen=True)
class LspShape:
    name: str
    C: int          # concurrency (requests per round)
    B: int          # draft block slots (= proposals per round)
    L: int          # tapped target layers
    D: int          # drafter layers
    H: int          # hidden size
    nq: int         # query heads
    nkv: int        # key/value heads
    d: int          # head dim
    F: int          # MLP width
    V: int          # vocabulary
    W: int = 256    # recent window rows per tapped layer (App. B.1)
    R: int = 16     # summary queries per tapped layer and head (App. B.1)
    rc: int = 64    # rank of the Markov correction
    dtype: str = "bf16"
    prefix: int = 0                 # prefix length folded into the state
    prefixes: tuple = ()            # prefix sweep (when non-empty)
    temperature: float = 0.0        # 0 = greedy
    rope_theta: float = 1.0e6
    rms_eps: float = 1.0e-6
    layer_scale: bool = False       # per-layer RMS scale U[0.5, 2] on K, V, h
    outlier_frac: float = 0.0       # fraction of channels scaled by outlier_mult
    outlier_mult: float = 1.0
    delta_max: int = 16             # accepted_len ~ U[1, delta_max]
    layer_map: tuple = ()           # draft layer j -> tapped index (default floor(j*L/D))
    no_boundary: bool = False       # ablation: no boundary state / fusion (W = 0, R = 0: the others)

    def __post_init__(self):
        if not self.layer_map:
            object.__setattr__(self, "layer_map",
                               tuple(j * self.L // self.D for j in range(self.D)))

    @property
    def M(self) -> int:
        return self.C * self.B

    @property
    def torch_dtype(self):
        return torch.bfloat16 if self.dtype == "bf16" else torch.float32

    def with_(self, **kw) -> "LspShape":
        kw.setdefault("layer_map", ())
        return dataclasses.replace(self, **kw)


# The five workload shapes (draft block = B, tapped layers = L, drafter depth = D).
TINY = LspShape("tiny", C=1, B=8, L=3, D=1, H=256, nq=4, nkv=2, d=64, F=1024, V=1024,
                dtype="f32", prefix=2048, temperature=0.0, delta_max=8)
SMALL = LspShape("small", C=4, B=16, L=4, D=2, H=1024, nq=8, nkv=2, d=128, F=4096,
                 V=32000, prefix=8192, temperature=0.0, layer_scale=True)
Q8B = LspShape("qwen3-8b", C=16, B=16, L=5, D=5, H=4096, nq=32, nkv=8, d=128, F=12288,
               V=151936, prefix=32768, temperature=1.0)
SWEEP = Q8B.with_(name="qwen3-8b-sweep", prefixes=(4096, 16384, 65536, 131072))
LARGE = LspShape("large", C=32, B=16, L=5, D=5, H=5120, nq=40, nkv=8, d=128, F=17408,
                 V=151936, prefix=131072, temperature=1.0, outlier_frac=0.01,
                 outlier_mult=20.0)

SHAPES = {s.name: s for s in (TINY, SMALL, Q8B, SWEEP, LARGE)}

WEIGHT_SEED = 42
RNG_SEED = 7


def input_seed(shape: LspShape) -> int:
    return 1234 + list(SHAPES).index(shape.name) if shape.name in SHAPES else 1234


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def _normal(shape, std, g, device, dtype):
    t = torch.randn(*shape, generator=g, device=device, dtype=torch.float32)
    if std != 1.0:
        t.mul_(std)
    return t.to(dtype)


def make_weights(shape: LspShape, seed: int = WEIGHT_SEED, device="cpu") -> dict:
    """Random-init drafter weights in the layout the C ABI documents.

    Linear weights are [out_features][in_features] (row-major, in contiguous).
    """
    s, dt = shape, shape.torch_dtype
    g = _gen(seed, device)
    std = 0.02

    def lin(o, i):
        return _normal((o, i), std, g, device, dt)

    def norm(n):
        return (1.0 + 0.1 * torch.randn(n, generator=g, device=device)).to(dt)

    w = {
        "embed": lin(s.V, s.H),
        "final_norm": norm(s.H),
        "lm_head": lin(s.V, s.H),
        "fuse": lin(s.H, s.L * s.H),
        "pos": lin(s.B, s.H),
        "mask_emb": _normal((s.H,), std, g, device, dt),
        "G": _normal((s.L, s.nq, s.R, s.d), (1.0 / s.d) ** 0.5, g, device, dt),
        "Ec": lin(s.V, s.rc),
        "Wc": lin(s.V, s.rc),
        "layers": [],
    }
    for _ in range(s.D):
        w["layers"].append({
            "in_norm": norm(s.H),
            "wq": lin(s.nq * s.d, s.H),
            "wk": lin(s.nkv * s.d, s.H),
            "wv": lin(s.nkv * s.d, s.H),
            "q_norm": norm(s.d),
            "k_norm": norm(s.d),
            "wo": lin(s.H, s.nq * s.d),
            "post_norm": norm(s.H),
            "w_gate": lin(s.F, s.H),
            "w_up": lin(s.F, s.H),
            "w_down": lin(s.H, s.F),
        })
    return w


def _feature_scales(shape: LspShape, device):
    """Per-layer RMS scales and outlier-channel multipliers (fixed per shape)."""
    g = _gen(9000 + input_seed(shape), "cpu")
    if shape.layer_scale:
        lsc = 0.5 + 1.5 * torch.rand(shape.L, generator=g)
    else:
        lsc = torch.ones(shape.L)
    kv_mult = torch.ones(shape.nkv * shape.d)
    h_mult = torch.ones(shape.H)
    if shape.outlier_frac > 0:
        nk = max(1, int(round(shape.outlier_frac * kv_mult.numel())))
        nh = max(1, int(round(shape.outlier_frac * h_mult.numel())))
        kv_mult[torch.randperm(kv_mult.numel(), generator=g)[:nk]] = shape.outlier_mult
        h_mult[torch.randperm(h_mult.numel(), generator=g)[:nh]] = shape.outlier_mult
    return lsc.to(device), kv_mult.to(device), h_mult.to(device)


def make_features(shape: LspShape, n_rows: int, seed: int, device="cpu", with_h=True):
    """Target features for `n_rows` new rows per request and tapped layer.

    Returns (k, v, h): k, v are [C][L][n_rows][nkv][d]; h is [C][L][n_rows][H]
    (or None when with_h is False), all in the shape's storage dtype.
    """
    s, dt = shape, shape.torch_dtype
    g = _gen(seed, device)
    lsc, kv_mult, h_mult = _feature_scales(s, device)
    k = torch.randn(s.C, s.L, n_rows, s.nkv * s.d, generator=g, device=device)
    v = torch.randn(s.C, s.L, n_rows, s.nkv * s.d, generator=g, device=device)
    sc = lsc.view(1, s.L, 1, 1) * kv_mult.view(1, 1, 1, -1)
    k = (k * sc).to(dt).view(s.C, s.L, n_rows, s.nkv, s.d)
    v = (v * sc).to(dt).view(s.C, s.L, n_rows, s.nkv, s.d)
    h = None
    if with_h:
        h = torch.randn(s.C, s.L, n_rows, s.H, generator=g, device=device)
        h = (h * (lsc.view(1, s.L, 1, 1) * h_mult.view(1, 1, 1, -1))).to(dt)
    return k, v, h


def make_accepted(shape: LspShape, seed: int, device="cpu", lo: int = 1, hi: int | None = None):
    """accepted_len per request: U[lo, hi] (default hi = delta_max), int32 [C]."""
    hi = shape.delta_max if hi is None else hi
    g = _gen(seed, "cpu")
    return torch.randint(lo, hi + 1, (shape.C,), generator=g, dtype=torch.int32).to(device)


def make_block_tokens(shape: LspShape, seed: int, device="cpu"):
    """int32 [C][B]: slot 0 holds the committed token a ~ U[0, V); the others are -1 (mask)."""
    g = _gen(seed, "cpu")
    bt = torch.full((shape.C, shape.B), -1, dtype=torch.int32)
    bt[:, 0] = torch.randint(0, shape.V, (shape.C,), generator=g, dtype=torch.int32)
    return bt.to(device)


def make_verify_logits(shape: LspShape, seed: int, std: float = 2.0, agree=(0.9, 0.999)):
    """Target and draft logits of one verification call, fp32.

    zt [C][B+1][V] ~ N(0, std^2); the draft row i of request b is
    a_b zt[b, i] + sqrt(1 - a_b^2) N(0, std^2) with a_b ~ U[agree]: requests range
    from a drafter that mostly agrees with the target to one that often does not,
    so the accepted lengths spread over [0, B].
    """
    g = _gen(seed, "cpu")
    C, B, V = shape.C, shape.B, shape.V
    zt = torch.randn((C, B + 1, V), generator=g, dtype=torch.float32) * std
    a = agree[0] + (agree[1] - agree[0]) * torch.rand((C, 1, 1), generator=g, dtype=torch.float64)
    noise = torch.randn((C, B, V), generator=g, dtype=torch.float32) * std
    zq = (a * zt[:, :B].double() + torch.sqrt(1 - a * a) * noise.double()).float()
    return zt.contiguous(), zq.contiguous()
