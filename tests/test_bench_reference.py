"""bench.py's reference arm (the oracle on the host cores) end to end on CPU: the
tiny shape with the generators on the host; it prints the contract's JSON line,
with exactly `steps` whole rounds timed after `warmup` untimed ones, without
loading or running the library."""
import argparse
import json
import os
import sys

import numpy as np
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_prints_the_oracle_line(capsys):
    sys.path.insert(0, ROOT)
    import bench
    args = argparse.Namespace(config="tiny", prefix=300, steps=2, warmup=1, cpu_budget=30.0, gpus=1)

    class OneRank:
        rank, world = 0, 1

    loaded_before = "paper_2609_37029_gb300.lsp" in sys.modules
    bench.run_reference(args, OneRank(), device="cpu")
    line = [l for l in capsys.readouterr().out.splitlines() if l.startswith("{")][-1]
    out = json.loads(line)
    assert out["impl"] == "reference" and out["unit"] == bench.UNIT and out["metric"] == bench.METRIC
    assert out["value"] > 0 and out["higher_is_better"] is True and out["dtype"] == "f64"
    assert out["steps"] == 2 and out["warmup"] == 1            # the rounds actually timed
    assert out["value"] * out["ms_per_step"] * 1e-3 == __import__("pytest").approx(1 * 8)   # C x B per round
    assert out["cpu_baseline"]["kind"] == "oracle" and out["cpu_baseline"]["value"] == out["value"]
    assert out["e2e"] == {"value": out["value"], "unit": out["unit"], "h2d_bytes_per_step": 0,
                          "d2h_bytes_per_step": 0}
    assert out["config"]["workload"].startswith("tiny drafting round")
    if not loaded_before:                     # the oracle's arm never touched the library
        assert "paper_2609_37029_gb300.lsp" not in sys.modules


def test_oracle_fold_takes_the_seeded_chunks_the_library_folds():
    """The oracle's prefix is the same seeded chunks fold() hands the library: after
    FOLD_CHUNK + 5 rows the window holds the last W rows of those chunks and the boundary
    is the last row of the shared hidden-state chunk."""
    sys.path.insert(0, ROOT)
    import bench
    import oracle
    from paper_2609_37029_gb300 import synth
    s = synth.SHAPES["tiny"].with_(C=2)
    wl = bench.Workload(s, None, 123, device="cpu")
    so = s.with_(C=1)
    ost = oracle.state_init(so)
    G = np.zeros((s.L, s.nq, s.R, s.d))
    n = bench.FOLD_CHUNK + 5
    wl.oracle_fold(so, ost, G, 0, n, [1])
    assert list(ost.t) == [n]
    k0, _, _ = synth.make_features(s, bench.FOLD_CHUNK, seed=123, device="cpu", with_h=False)
    k1, _, _ = synth.make_features(s, bench.FOLD_CHUNK, seed=123 + 1, device="cpu", with_h=False)
    _, _, h = synth.make_features(s, bench.FOLD_CHUNK, seed=123 + 7000, device="cpu")
    want = torch.cat([k0[1, :, bench.FOLD_CHUNK - (s.W - 5):], k1[1, :, :5]], dim=1).double().numpy()
    for l in range(s.L):
        assert np.array_equal(ost.win_k[0][l], want[l])
    assert np.array_equal(ost.hb[0], h[1, :, 4].double().numpy())
