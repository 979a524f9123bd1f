#!/usr/bin/env python
"""Benchmark of the fixed-cost drafting round on one GB300 (or N replicas).

One step = one drafting round over all C requests: lsp_view_update (fold the
new target rows into the fixed-size interface) + lsp_draft (boundary fusion,
D draft layers, LM head, Markov correction + sampling of B proposals).

Default workload: Qwen3-8B-shaped drafter at concurrency 16, 32K-token prefix,
temperature-1 sampling (C=16, B=16, L=5 tapped layers, D=5, H=4096, 32 q / 8 kv
heads x 128, MLP 12288, V=151936, W=256, R=16).  All inputs are seeded
synthetic tensors (see paper_2609_37029_gb300/synth.py); weights are random
init.  The 3.3 GB of projection weights streamed every round exceed the
129 MB L2, so no explicit flush is needed between timed rounds.

Prints one JSON line (rank 0).  `--impl reference` times the fp64 oracle on
the host cores instead (the reference arm: there is no other implementation
of the method to run).  `--profile-rounds N` only folds the prefix and runs N
eager rounds, for a profiler.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np
import torch

from paper_2609_37029_gb300 import synth

METRIC = "drafting µs/round and drafted tokens/s vs prefix length at concurrency 16; % roofline"
UNIT = "drafted tokens/s"
FOLD_CHUNK = 2048
GEMM_STAGES = ("fuse", "qkv", "o_proj", "gate_up", "down", "lm_head")


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=50)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default="qwen3-8b", choices=sorted(synth.SHAPES))
    ap.add_argument("--prefix", type=int, default=None)
    ap.add_argument("--no-sweep", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--cpu-budget", type=float, default=150.0, help="seconds for the oracle legs")
    ap.add_argument("--profile-rounds", type=int, default=0,
                    help="only fold the prefix and run this many eager rounds, then exit "
                         "(a short, untimed command for a profiler)")
    return ap.parse_args()


# ------------------------------------------------------------------ distributed plumbing
class Dist:
    """One process per GPU (torchrun env); replicas only: the ranks share no data,
    only the barrier around the timed region and the max of the ranks' times.
    Backend nccl on GPUs, gloo otherwise (or LSP_DIST_BACKEND)."""

    def __init__(self, backend=None):
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local = int(os.environ.get("LOCAL_RANK", "0"))
        self.pg = None
        self.device = "cpu"
        if self.world > 1:
            import torch.distributed as dist
            backend = backend or os.environ.get("LSP_DIST_BACKEND") or (
                "nccl" if torch.cuda.is_available() else "gloo")
            if backend == "nccl":
                torch.cuda.set_device(self.local)
                self.device = f"cuda:{self.local}"
                dist.init_process_group("nccl", device_id=torch.device("cuda", self.local))
            else:
                dist.init_process_group(backend)
            self.pg = dist

    def barrier(self):
        if self.pg:
            self.pg.barrier()

    def max(self, x: float) -> float:
        if not self.pg:
            return x
        t = torch.tensor([x], device=self.device, dtype=torch.float64)
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX)
        return float(t.item())

    def close(self):
        if self.pg:
            self.pg.destroy_process_group()


def job_throughput(world: int, C: int, B: int, ms: float) -> float:
    """Whole-job drafted tokens/s: every replica drafts C x B tokens per round; `ms`
    is the max over ranks of the per-round time (weak scaling)."""
    return world * C * B / (ms * 1e-3)


# ------------------------------------------------------------------ clocks during the timed region
class Clocks:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self):
        self.proc = None
        self.target = self._gpu_id()

    @staticmethod
    def _gpu_id():
        try:
            p = torch.cuda.get_device_properties(torch.cuda.current_device())
            return f"{p.pci_domain_id:08X}:{p.pci_bus_id:02X}:{p.pci_device_id:02X}.0"
        except Exception:
            vis = os.environ.get("CUDA_VISIBLE_DEVICES", "0").split(",")[0]
            return vis or "0"

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.target}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"]}
        self.proc.terminate()
        try:
            out = self.proc.communicate(timeout=10)[0]
        except Exception:
            self.proc.kill()
            out = ""
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "samples": len(sm), "reasons": sorted(reasons)}


# ------------------------------------------------------------------ algorithmic work
def gemm_work(s, name):
    """(bytes, flops) of one projection launch: weights + activations in + outputs out."""
    es = 2 if s.dtype == "bf16" else 4
    M = s.C * s.B
    if name == "fuse":
        Mx, N, K, out = s.C, s.H, s.L * s.H, s.C * s.H * 4
    elif name == "qkv":
        Mx, N, K = M, (s.nq + 2 * s.nkv) * s.d, s.H
        out = M * N * es
    elif name == "o_proj":
        Mx, N, K = M, s.H, s.nq * s.d
        out = 2 * M * N * 4                      # residual read + write
    elif name == "gate_up":
        Mx, N, K = M, 2 * s.F, s.H
        out = M * s.F * es
    elif name == "down":
        Mx, N, K = M, s.H, s.F
        out = 2 * M * N * 4
    else:                                        # lm_head
        Mx, N, K = M, s.V, s.H
        out = M * N * 4
    return N * K * es + Mx * K * es + out, 2.0 * Mx * N * K


def round_work(s, mean_delta):
    """Algorithmic bytes / flops of one round: weights once, interface state touched, one logits write."""
    es = 2 if s.dtype == "bf16" else 4
    nb = 0
    fl = 0.0
    names = ["fuse"] + ["qkv", "o_proj", "gate_up", "down"] * s.D + ["lm_head"]
    for n in names:
        b, f = gemm_work(s, n)
        nb += b
        fl += f
    kv = s.nkv * s.d
    # view update: new K/V rows read + window write, summary (m, eta) read+write, G, boundary
    nb += s.C * mean_delta * s.L * 2 * kv * es * 2
    nb += 2 * s.C * s.L * s.nq * s.R * (s.d + 1) * 4 + s.L * s.nq * s.R * s.d * es + s.C * s.L * s.H * es
    fl += 4.0 * s.C * s.L * s.nq * s.R * mean_delta * s.d
    # attention: window K/V + summary values per draft layer
    ctx = s.B + s.W + s.R
    nb += s.C * s.D * (s.W * 2 * kv * es + s.nq * s.R * s.d * 4)
    fl += 4.0 * s.C * s.D * s.nq * s.B * ctx * s.d
    # correction factors and the sampler's corrected-logit pass
    nb += 2 * s.V * s.rc * es
    fl += 2.0 * s.C * s.B * s.V * s.rc
    return nb, fl


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            j = json.load(f)
        return float(j["hbm_gbs"]), float(j["bf16_tflops"]), float(j["bf16_tflops_sustained"]), "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


def profiled_traffic(kernel_file, workload):
    """DRAM bytes per launch from a committed ncu summary, if taken on the current source."""
    path = os.path.join(ROOT, "profiles", f"{kernel_file}_{workload}.md")
    src = os.path.join(ROOT, "paper_2609_37029_gb300", "csrc", kernel_file.split("__")[0] + ".cu")
    try:
        sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
        txt = open(path).read()
    except OSError:
        return None
    vals = {}
    for line in txt.splitlines():
        if line.startswith("traffic_key:"):
            k, v = line.split(":", 1)[1].split("=")
            vals[k.strip()] = v.strip()
    if vals.get("source_sha256_16") != sha:
        return None
    try:
        return float(vals["dram_bytes_per_round"])
    except (KeyError, ValueError):
        return None


def prefill_leg(wl, rows, hbm, dist, reps=5):
    """lsp_prefill of one request's `rows`-row prefix: device time, K/V bytes read, HBM fraction."""
    s, lsp = wl.s, wl.lsp
    s1 = s.with_(C=1)
    k, v, h = synth.make_features(s1, rows, seed=wl.seed_base + 9000, device="cuda")
    st = wl.new_state()
    for _ in range(2):
        lsp.lsp_prefill(st, 0, k[0], v[0], h[0])
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    dist.barrier()
    e0.record()
    for _ in range(reps):
        lsp.lsp_prefill(st, 0, k[0], v[0], h[0])
    e1.record()
    torch.cuda.synchronize()
    us = dist.max(e0.elapsed_time(e1) * 1e3 / reps)
    kv = 2 * s.L * rows * s.nkv * s.d * 2
    flops = 2 * 2 * s.L * s.nq * s.R * rows * s.d           # G K^T and P V
    lsp.lsp_state_destroy(st)
    del k, v, h
    return {"rows": rows, "us_per_request": us, "kv_bytes": kv, "achieved_gbs": kv / us * 1e-3,
            "frac_hbm": kv / us * 1e-3 / hbm, "flops": flops,
            "note": "mma.sync score and value products (P V as bf16 high + remainder): "
                    "tensor-issue bound on the legacy path, not HBM"}


def verify_leg(wl, hbm, dist, reps=20):
    """lsp_verify of one round's blocks against (synthetic) target logits [C][B+1][V]:
    device time and HBM fraction at T = 1 (residual / bonus draws) and T = 0 (greedy)."""
    s, lsp = wl.s, wl.lsp
    zt, _ = synth.make_verify_logits(s, seed=wl.seed_base + 9500)
    zt = zt.cuda()
    acc = torch.zeros(s.C, dtype=torch.int32, device="cuda")
    tok = torch.zeros(s.C, dtype=torch.int32, device="cuda")
    st = wl.new_state()
    out = {"C": s.C, "B": s.B, "V": s.V}
    for name, T in (("T1", 1.0), ("T0", 0.0)):
        sp = lsp.make_sample_params(T, seed=synth.RNG_SEED, rnd=1)
        for _ in range(3):
            lsp.lsp_verify(st, zt, wl.logits, wl.toks, sp, acc, tok)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        dist.barrier()
        e0.record()
        for _ in range(reps):
            lsp.lsp_verify(st, zt, wl.logits, wl.toks, sp, acc, tok)
        e1.record()
        torch.cuda.synchronize()
        us = dist.max(e0.elapsed_time(e1) * 1e3 / reps)
        # every row read once for its statistics, plus the emitting rows re-read by the draw
        rows = s.C * (2 * s.B + 3) if T > 0 else s.C * (s.B + 1)
        nbytes = rows * s.V * 4
        out[name] = {"us": us, "bytes": nbytes, "achieved_gbs": nbytes / us * 1e-3,
                     "frac_hbm": nbytes / us * 1e-3 / hbm}
    assert lsp.lsp_get_error(st) == (lsp.LSP_OK, 0)
    lsp.lsp_state_destroy(st)
    out["note"] = ("inputs %.0f MB > L2 (no flush needed); T = 1 reads target and draft rows, "
                   "T = 0 the target rows only" % (s.C * (2 * s.B + 1) * s.V * 4 / 1e6))
    return out


def variants_leg(s, lsp, seed_base, dist, steps=100, prefix=4096):
    """Round time of the paper's B = 7 and of the three ablation variants (Sec. 3.4) on
    the same kernels: drafted tokens/s and the per-request interface bytes."""
    out = {}
    for name, kw in (("B7", {"B": 7}), ("no_window", {"W": 0}), ("no_summary", {"R": 0}),
                     ("no_boundary", {"no_boundary": True})):
        sv = s.with_(**kw)
        wl = Workload(sv, lsp, seed_base + 300)
        st = wl.new_state()
        wl.fold(st, 0, prefix)
        for _ in range(2):
            wl.round(st)
        g = wl.capture(st)
        ms, _ = time_graph(g, steps, 10, dist)
        ms = dist.max(ms)
        assert lsp.lsp_get_error(st) == (lsp.LSP_OK, 0)
        out[name] = {"us_per_round": ms * 1e3, "drafted_tokens_per_s": dist.world * sv.C * sv.B / (ms * 1e-3),
                     "state_bytes": lsp.lsp_state_bytes(wl.cfg), "launches": lsp.lsp_round_launches(st)}
        del g
        lsp.lsp_state_destroy(st)
        del wl
        torch.cuda.empty_cache()
    out["note"] = "prefix %d rows folded; same weights recipe; W = 0 / R = 0 / no boundary remove one context source" % prefix
    return out


# ------------------------------------------------------------------ workload
class Workload:
    """Seeded synthetic inputs of one shape (weights, a round's new rows, accepted
    lengths, block tokens, prefix chunks) and, given the library binding `lsp`, the
    round driven through it.  Without `lsp` (the oracle's arm) nothing of the
    library is loaded; `device` is where the generators run (CUDA for both arms,
    so that they see the same values)."""

    def __init__(self, s, lsp, seed_base, device="cuda"):
        self.s, self.lsp = s, lsp
        self.seed_base = seed_base
        self.device = device
        self.w = synth.make_weights(s, seed=synth.WEIGHT_SEED, device=device)
        rows = s.B + 1
        self.k, self.v, self.h = synth.make_features(s, rows, seed=seed_base + 5000, device=device)
        self.acc = synth.make_accepted(s, seed=seed_base + 5001, device=device, hi=min(s.delta_max, s.B + 1))
        self.bt = synth.make_block_tokens(s, seed=seed_base + 5002, device=device)
        self._hfold = None
        if lsp is not None:
            self.ws = lsp.make_weights(self.w)
            self.cfg = lsp.make_config(s)
            self.toks = torch.zeros(s.C, s.B, dtype=torch.int32, device=device)
            self.logits = torch.empty(s.C, s.B, s.V, device=device)
            self.sp = lsp.make_sample_params(s.temperature, seed=synth.RNG_SEED, rnd=0)

    def new_state(self):
        st = self.lsp.lsp_state_create(self.cfg)
        self.lsp.lsp_state_init(st, self.w["G"])
        return st

    def _chunks(self, start, end):
        """Prefix rows [start, end) as seeded FOLD_CHUNK-row chunks: (k, v, h, rows used)."""
        s = self.s
        if self._hfold is None:
            _, _, self._hfold = synth.make_features(s, FOLD_CHUNK, seed=self.seed_base + 7000,
                                                    device=self.device)
        for c0 in range(start, end, FOLD_CHUNK):
            k, v, _ = synth.make_features(s, FOLD_CHUNK, seed=self.seed_base + c0 // FOLD_CHUNK,
                                          device=self.device, with_h=False)
            yield k, v, self._hfold, min(FOLD_CHUNK, end - c0)

    def fold(self, st, start, end):
        """Fold prefix rows [start, end) into `st` through the library, chunk by chunk."""
        for k, v, h, n in self._chunks(start, end):
            acc = torch.full((self.s.C,), n, dtype=torch.int32, device=self.device)
            self.lsp.lsp_view_update(st, k, v, h, acc, rows=FOLD_CHUNK)

    def oracle_fold(self, so, ost, G, start, end, reqs):
        """Fold the same prefix rows [start, end) of requests `reqs` into the oracle state
        `ost` (oracle shape `so`, C = len(reqs)); nothing runs in the library.  Only each
        chunk's last hidden row enters the boundary, so only that row is converted."""
        import oracle
        s = self.s
        for k, v, h, n in self._chunks(start, end):
            kk = k[reqs][:, :, :n].to(torch.float64).cpu().numpy()
            vv = v[reqs][:, :, :n].to(torch.float64).cpu().numpy()
            hl = np.broadcast_to(h[reqs][:, :, n - 1:n].to(torch.float64).cpu().numpy(),
                                 (len(reqs), s.L, n, s.H))
            oracle.view_update(so, ost, G, kk, vv, hl, np.full(len(reqs), n))

    def round(self, st):
        self.lsp.lsp_view_update(st, self.k, self.v, self.h, self.acc)
        self.lsp.lsp_draft(st, self.bt, self.ws, self.sp, self.toks, self.logits)

    def capture(self, st):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.round(st)
        return g


def round_percentiles(g, n=200):
    """Per-round device times of n replays, each between its own pair of CUDA
    events (after the main timed region): median, p10, p90 in µs."""
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(n + 1)]
    torch.cuda.synchronize()
    evs[0].record()
    for i in range(n):
        g.replay()
        evs[i + 1].record()
    torch.cuda.synchronize()
    t = sorted(evs[i].elapsed_time(evs[i + 1]) * 1e3 for i in range(n))
    return {"median": t[n // 2], "p10": t[n // 10], "p90": t[(9 * n) // 10], "n": n}


def time_graph(g, steps, warmup, dist, clocks=None):
    if clocks:
        clocks.start()                  # samples span the warm-up and the timed replays
    for _ in range(warmup):
        g.replay()
    torch.cuda.synchronize()
    dist.barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(steps):
        g.replay()
    e1.record()
    torch.cuda.synchronize()
    dist.barrier()
    ck = clocks.stop() if clocks else None
    return e0.elapsed_time(e1) / steps, ck


def stage_times(wl, st, reps):
    """Per-stage device time of a captured round via the library's stage-event hook."""
    lsp = wl.lsp
    n = lsp.lsp_stage_count(st)
    names = [lsp.lsp_stage_name(st, k) for k in range(n)]
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(n + 1)]
    for e in evs:
        e.record()
    torch.cuda.synchronize()
    lsp.lsp_set_stage_events(st, evs)
    try:
        g = wl.capture(st)
        run = g.replay
    except Exception:                    # event nodes not capturable here: time eager rounds
        g = None
        run = lambda: wl.round(st)
    acc = np.zeros(n)
    try:
        for _ in range(3):
            run()
        torch.cuda.synchronize()
        for _ in range(reps):
            run()
            torch.cuda.synchronize()
            acc += [evs[k].elapsed_time(evs[k + 1]) for k in range(n)]
    finally:
        lsp.lsp_set_stage_events(st, [])
    return names, acc / reps


# ------------------------------------------------------------------ oracle (CPU) legs
def oracle_weights(w):
    import oracle

    def host64(t):
        return t.detach().to(torch.float64).cpu().numpy()

    wn = {k: host64(v) for k, v in w.items() if k not in ("layers", "embed")}
    wn["embed"] = w["embed"].detach().float().cpu().numpy()       # rows gathered on use
    wn["layers"] = [{k: host64(v) for k, v in lw.items()} for lw in w["layers"]]
    return oracle.OracleWeights(wn)


class OracleRound:
    """One whole drafting round of all C requests as the oracle computes it (view update of
    the round's new rows, drafter forward, B-step correction + sampling per request), on
    the state the same seeded prefix gives.  The round's inputs are converted to fp64 on
    the host once, outside the timed calls."""

    def __init__(self, wl, prefix):
        import oracle
        s = wl.s
        self.s, self.wl = s, wl
        self.reqs = list(range(s.C))
        self.ow = oracle_weights(wl.w)
        self.ost = oracle.state_init(s)
        wl.oracle_fold(s, self.ost, self.ow.G, 0, prefix, self.reqs)
        f64 = lambda t: t.detach().to(torch.float64).cpu().numpy()
        self.k, self.v, self.h = f64(wl.k), f64(wl.v), f64(wl.h)
        self.acc = wl.acc.cpu().numpy()
        self.bt = wl.bt.cpu().numpy()

    def step(self):
        """One round; returns its wall-clock seconds."""
        import oracle
        s, ow, ost = self.s, self.ow, self.ost
        t0 = time.perf_counter()
        oracle.view_update(s, ost, ow.G, self.k, self.v, self.h, self.acc)
        z0 = oracle.draft_base_logits(s, ost, ow, self.bt)
        for b in self.reqs:
            oracle.sample_block(z0[b], int(self.bt[b, 0]), ow.Ec, ow.Wc, s.temperature, synth.RNG_SEED, 0, b)
        return time.perf_counter() - t0


def host_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def blas_threads():
    for var in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        if os.environ.get(var):
            return int(os.environ[var])
    return host_cores()


CPU_PREFIX = 4096          # prefix rows the in-run CPU baseline folds (the round's cost is prefix-free)


def oracle_leg(wl, budget, prefix=CPU_PREFIX, warmup=1, min_s=10.0):
    """The in-run CPU baseline: whole rounds of all C requests on the host cores after a
    `prefix`-row prefix (the state is fixed-size, so a round costs the same at any prefix),
    one warm-up round, then rounds until `min_s` seconds of them (or `budget`) are timed."""
    s = wl.s
    orr = OracleRound(wl, prefix)
    for _ in range(warmup):
        orr.step()
    times = []
    while not times or (sum(times) < min_s and sum(times) < budget):
        times.append(orr.step())
    t_round = statistics.mean(times)
    return {"value": s.C * s.B / t_round, "unit": UNIT, "cores": host_cores(), "blas_threads": blas_threads(),
            "kind": "oracle",
            "sample": (f"{len(times)} whole round(s) of all {s.C} requests (view update of the round's "
                       f"new rows, drafter forward, {s.B}-step correction + sampling) in numpy fp64 after "
                       f"{warmup} warm-up, on the state of a {prefix}-row prefix; mean {t_round:.2f} s per round"),
            "_t_round": t_round, "_steps": len(times)}


# ------------------------------------------------------------------ main
def workload_config(s, prefix):
    return {"workload": (f"{s.name} drafting round: C={s.C}, B={s.B}, {s.L} tapped layers, D={s.D}, "
                         f"H={s.H}, {s.nq}q/{s.nkv}kv x {s.d}, F={s.F}, V={s.V}, W={s.W}, R={s.R}, "
                         f"r_c={s.rc}, prefix {prefix}, "
                         + ("greedy" if s.temperature == 0 else f"T={s.temperature:g} sampling")),
            "C": s.C, "B": s.B, "prefix": prefix, "global_batch": s.C, "seq_len": prefix,
            "parallelism": "replicas", "accepted_len": f"U[1,{s.delta_max}] seeded",
            "l2": "no flush: >3 GB of weights streamed per round exceed the 129 MB L2"}


def run_reference(args, dist, device="cuda"):
    """The oracle's arm: the same seeded inputs and prefix, whole rounds of all C requests
    by the oracle alone on the host cores (the library is neither loaded nor run):
    `warmup` untimed rounds, then `steps` timed rounds."""
    if dist.rank != 0:
        return
    s = synth.SHAPES[args.config]
    prefix = args.prefix or s.prefix
    wl = Workload(s, None, synth.input_seed(s) * 1000, device=device)
    orr = OracleRound(wl, prefix)
    for _ in range(args.warmup):
        orr.step()
    times = [orr.step() for _ in range(max(1, args.steps))]
    t_round = statistics.mean(times)
    ms = t_round * 1e3
    value = s.C * s.B / t_round
    out = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
           "n_gpus": args.gpus, "steps": len(times), "warmup": args.warmup,
           "ms_per_step": ms, "us_per_round": ms * 1e3, "higher_is_better": True, "scaling": "weak",
           "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": workload_config(s, prefix),
           "cpu_baseline": {"value": value, "unit": UNIT, "cores": host_cores(), "blas_threads": blas_threads(),
                            "kind": "oracle",
                            "sample": (f"{len(times)} whole rounds of all {s.C} requests after {args.warmup} "
                                       f"warm-up, on the state of the {prefix}-row prefix")},
           "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
           "note": "each step is one whole round of all requests by the fp64 oracle on the host cores"}
    print(json.dumps(out), flush=True)


def gemm_roofline(s, names, st_ms, hbm, tf_burst, tf_sust, peak_src, traffic_round=None):
    """The projection GEMM's algorithmic bytes and flops over its stage times."""
    gemm_bytes = gemm_flops = gemm_ms = 0.0
    for n, t in zip(names, st_ms):
        if n in GEMM_STAGES:
            b, f = gemm_work(s, n)
            gemm_bytes += b
            gemm_flops += f
            gemm_ms += float(t)
    n_gemm = sum(1 for n in names if n in GEMM_STAGES and (n != "fuse" or not s.no_boundary))
    ach = gemm_bytes / (gemm_ms * 1e-3) / 1e9
    intensity = gemm_flops / gemm_bytes
    ridge = tf_burst * 1e12 / (hbm * 1e9)
    tflops = gemm_flops / (gemm_ms * 1e-3) / 1e12
    return {"bound": "hbm" if intensity < ridge else "tensor",
            "kernel": f"gemm_kernel (tcgen05 projection GEMM, {n_gemm} launches per round)",
            "achieved": ach, "peak": hbm, "unit": "GB/s", "frac": ach / hbm,
            "peak_source": f"{peak_src} HBM copy bandwidth",
            "traffic": (traffic_round / n_gemm) if traffic_round else None,
            "algorithmic_bytes_per_launch": gemm_bytes / n_gemm,
            "avg_launch_us": gemm_ms * 1e3 / n_gemm,
            "tensor_tflops": tflops,
            "tensor_frac_of_burst": tflops / tf_burst,
            "tensor_frac_of_sustained": tflops / tf_sust,
            "intensity_flop_per_byte": intensity}


def round_roofline(s, ms, mean_delta, hbm, tf_burst):
    rb, rf = round_work(s, mean_delta)
    t_b, t_f = rb / (hbm * 1e9), rf / (tf_burst * 1e12)
    t_roof = max(t_b, t_f)
    return {"bytes": rb, "flops": rf, "bound": "hbm" if t_b >= t_f else "tensor",
            "roofline_us": t_roof * 1e6, "frac": t_roof * 1e3 / ms}


STAGES_NOTE = ("per-stage device time summed over the round's launches, from event records "
               "between stages (each ends the programmatic overlap at its boundary, so the stages "
               "sum to more than the round); 'qkv' is the q/k/v projection and 'attention' the "
               "tcgen05 attention with the q/k/v split sum, q/k norms and rotary folded in (shapes it "
               "does not serve run a separate finalize kernel inside 'qkv')")


def stage_dict(names, st_ms):
    stages = {}
    for n, t in zip(names, st_ms):
        stages[n] = stages.get(n, 0.0) + float(t) * 1e3
    return {k: round(v, 2) for k, v in stages.items()}


def configs_leg(lsp, dist, hbm, tf_burst, tf_sust, peak_src, steps=200, warmup=10):
    """The other workload shapes at their own prefixes on the same kernels: the fp32
    reference shape, the small bf16 shape, and the larger target (C = 32, 128K prefix,
    the tensor-bound one) sampled at T = 1 and greedy.  Per shape: device time per round
    (CUDA-graph replay), drafted tokens/s, the round's roofline, and the projection
    GEMM's HBM and tensor-pipe fractions from the per-stage events."""
    out = {}
    legs = (("tiny", "tiny", (None,)), ("small", "small", (None,)), ("large", "large", (1.0, 0.0)))
    for key, name, temps in legs:
        s0 = synth.SHAPES[name]
        wl = Workload(s0, lsp, synth.input_seed(s0) * 1000)
        st = wl.new_state()
        wl.fold(st, 0, s0.prefix)
        for T in temps:
            s = s0 if T is None else s0.with_(temperature=T)
            wl.s = s
            wl.sp = lsp.make_sample_params(s.temperature, seed=synth.RNG_SEED, rnd=0)
            for _ in range(2):
                wl.round(st)
            g = wl.capture(st)
            ms, _ = time_graph(g, steps, warmup, dist)
            ms = dist.max(ms)
            del g
            names, st_ms = stage_times(wl, st, reps=20)
            rc, bits = lsp.lsp_get_error(st)
            if rc != lsp.LSP_OK:
                raise RuntimeError(f"device error in the {name} leg: {rc} bits={bits}")
            mean_delta = float(wl.acc.float().mean())
            leg = {"workload": workload_config(s, s.prefix)["workload"], "C": s.C, "B": s.B,
                   "prefix": s.prefix, "temperature": s.temperature,
                   "us_per_round": ms * 1e3, "drafted_tokens_per_s": job_throughput(dist.world, s.C, s.B, ms),
                   "round_roofline": round_roofline(s, ms, mean_delta, hbm, tf_burst),
                   "gemm": {k: v for k, v in gemm_roofline(s, names, st_ms, hbm, tf_burst, tf_sust, peak_src).items()
                            if k in ("bound", "achieved", "frac", "tensor_tflops", "tensor_frac_of_burst",
                                     "tensor_frac_of_sustained", "avg_launch_us")},
                   "stages_us": stage_dict(names, st_ms), "launches": lsp.lsp_round_launches(st),
                   "dtype": s.dtype}
            out[key if T is None else f"{key}_{'T1' if T > 0 else 'greedy'}"] = leg
        lsp.lsp_state_destroy(st)
        del wl
        torch.cuda.empty_cache()
    return out


def run_ours(args, dist):
    from paper_2609_37029_gb300 import build as _b
    if dist.local == 0:
        _b.build()
    dist.barrier()
    from paper_2609_37029_gb300 import lsp
    torch.cuda.set_device(dist.local)
    s = synth.SHAPES[args.config]
    prefix = args.prefix or s.prefix
    hbm, tf_burst, tf_sust, peak_src = peaks()
    wl = Workload(s, lsp, synth.input_seed(s) * 1000)
    st = wl.new_state()
    want_cpu = dist.rank == 0 and dist.world == 1 and not args.no_cpu
    wl.fold(st, 0, prefix)
    for _ in range(2):
        wl.round(st)
    torch.cuda.synchronize()
    rc, bits = lsp.lsp_get_error(st)
    if rc != lsp.LSP_OK:
        raise RuntimeError(f"device error after warm-up: {rc} bits={bits}")
    g = wl.capture(st)
    ms, clocks = time_graph(g, args.steps, args.warmup, dist, Clocks())
    round_us = round_percentiles(g)
    ms = dist.max(ms)
    rc, bits = lsp.lsp_get_error(st)
    if rc != lsp.LSP_OK:
        raise RuntimeError(f"device error in the timed region: {rc} bits={bits}")

    # per-stage device times (dominant kernel = the projection GEMM)
    names, st_ms = stage_times(wl, st, reps=min(200, max(20, args.steps // 5)))
    roofline = gemm_roofline(s, names, st_ms, hbm, tf_burst, tf_sust, peak_src,
                             profiled_traffic("k_gemm", s.name))
    mean_delta = float(wl.acc.float().mean())
    round_roof = round_roofline(s, ms, mean_delta, hbm, tf_burst)

    # end to end through the C ABI with host buffers (pinned), copies inside the timed
    # region: the new K/V rows, each request's boundary hidden row (h_rows = 1: the only
    # row of h the view update reads), the accepted lengths and the block tokens in;
    # the drafted tokens out
    idx = (wl.acc.long().clamp(min=1) - 1).view(s.C, 1, 1, 1).expand(s.C, s.L, 1, s.H)
    h_last = torch.gather(wl.h, 2, idx).contiguous()
    hk, hv, hh = wl.k.cpu().pin_memory(), wl.v.cpu().pin_memory(), h_last.cpu().pin_memory()
    hacc, hbt = wl.acc.cpu().pin_memory(), wl.bt.cpu().pin_memory()
    htoks = torch.empty(s.C, s.B, dtype=torch.int32).pin_memory()

    def e2e_step():
        wl.k.copy_(hk, non_blocking=True)
        wl.v.copy_(hv, non_blocking=True)
        h_last.copy_(hh, non_blocking=True)
        wl.acc.copy_(hacc, non_blocking=True)
        wl.bt.copy_(hbt, non_blocking=True)
        lsp.lsp_view_update(st, wl.k, wl.v, h_last, wl.acc, rows=wl.k.shape[2], h_rows=1)
        lsp.lsp_draft(st, wl.bt, wl.ws, wl.sp, wl.toks, wl.logits)
        htoks.copy_(wl.toks, non_blocking=True)
        torch.cuda.current_stream().synchronize()

    k_e = min(args.steps, 300)
    for _ in range(min(args.warmup, 10)):
        e2e_step()
    dist.barrier()
    t0 = time.perf_counter()
    for _ in range(k_e):
        e2e_step()
    e2e_ms = dist.max((time.perf_counter() - t0) * 1e3 / k_e)
    h2d = sum(t.numel() * t.element_size() for t in (hk, hv, hh, hacc, hbt))
    d2h = htoks.numel() * htoks.element_size()

    # prefix sweep: drafting time and state bytes vs prefix length
    sweep = None
    prefixes = synth.SWEEP.prefixes if s.name in ("qwen3-8b", "qwen3-8b-sweep") else ()
    if prefixes and not args.no_sweep:
        st2 = wl.new_state()
        done = 0
        pts = {}
        for p in prefixes:
            wl.fold(st2, done, p)
            done = p
            g2 = wl.capture(st2)
            m2, _ = time_graph(g2, max(100, args.steps // 4), 10, dist)
            pts[str(p)] = dist.max(m2) * 1e3
            del g2
        vals = list(pts.values())
        sweep = {"us_per_round": pts, "max_over_min": max(vals) / min(vals),
                 "state_bytes": lsp.lsp_state_bytes(wl.cfg), "state_bytes_constant": True}
        lsp.lsp_state_destroy(st2)

    # prefill (the one O(t) drafter step): one request's whole prefix at the largest sweep length
    prefill = None
    if prefixes and not args.no_sweep and s.dtype == "bf16":
        prefill = prefill_leg(wl, max(prefixes), hbm, dist)

    verify = None
    if not args.no_sweep:
        verify = verify_leg(wl, hbm, dist)

    variants = None
    if not args.no_sweep and s.dtype == "bf16":
        variants = variants_leg(s, lsp, wl.seed_base, dist)

    configs = None
    if not args.no_sweep and s.name in ("qwen3-8b", "qwen3-8b-sweep"):
        configs = configs_leg(lsp, dist, hbm, tf_burst, tf_sust, peak_src)

    cpu = None
    if want_cpu:
        leg = oracle_leg(wl, args.cpu_budget)
        cpu = {k: v for k, v in leg.items() if not k.startswith("_")}

    value = job_throughput(dist.world, s.C, s.B, ms)
    out = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": dist.world,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "us_per_round": ms * 1e3,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if s.dtype == "bf16" else "f32",
           "round_us": round_us,
           "data": "synthetic (seeded random features and random-init weights)",
           "config": workload_config(s, prefix),
           "roofline": roofline, "round_roofline": round_roof,
           "stages_us": stage_dict(names, st_ms),
           "stages_note": STAGES_NOTE,
           "e2e": {"value": job_throughput(dist.world, s.C, s.B, e2e_ms), "unit": UNIT,
                   "ms_per_step": e2e_ms, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
           "gpu_launches": lsp.lsp_round_launches(st) * args.steps,
           "clocks": clocks, "sweep": sweep, "configs": configs, "prefill": prefill, "verify": verify,
           "variants": variants, "cpu_baseline": cpu}
    if dist.rank == 0:
        print(json.dumps(out), flush=True)
    lsp.lsp_state_destroy(st)


def profile_rounds(args):
    """Fold the prefix, run `--profile-rounds` eager rounds, check the device error
    word and exit: the launch sequence of a round without the timing legs."""
    from paper_2609_37029_gb300 import build as _b
    _b.build()
    from paper_2609_37029_gb300 import lsp
    s = synth.SHAPES[args.config]
    wl = Workload(s, lsp, synth.input_seed(s) * 1000)
    st = wl.new_state()
    wl.fold(st, 0, args.prefix or s.prefix)
    for _ in range(args.profile_rounds):
        wl.round(st)
    torch.cuda.synchronize()
    rc, bits = lsp.lsp_get_error(st)
    lsp.lsp_state_destroy(st)
    if rc != lsp.LSP_OK:
        raise RuntimeError(f"device error: {rc} bits={bits}")
    print(f"{args.profile_rounds} round(s) of {s.name} after a {args.prefix or s.prefix}-row prefix: ok")


def main():
    args = parse_args()
    if args.profile_rounds > 0:
        profile_rounds(args)
        return
    dist = Dist()
    try:
        if args.impl == "reference":
            run_reference(args, dist)
        else:
            run_ours(args, dist)
    finally:
        dist.close()


if __name__ == "__main__":
    main()
