"""bench.py's reference arm (the oracle on the host cores) end to end on CPU: the
tiny shape with the generators on the host, one step; it prints the contract's
JSON line without loading or running the library."""
import argparse
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_prints_the_oracle_line(capsys):
    sys.path.insert(0, ROOT)
    import bench
    args = argparse.Namespace(config="tiny", prefix=None, steps=1, warmup=1, cpu_budget=30.0, gpus=1)

    class OneRank:
        rank, world = 0, 1

    loaded_before = "paper_2609_37029_gb300.lsp" in sys.modules
    bench.run_reference(args, OneRank(), device="cpu")
    line = [l for l in capsys.readouterr().out.splitlines() if l.startswith("{")][-1]
    out = json.loads(line)
    assert out["impl"] == "reference" and out["unit"] == bench.UNIT and out["metric"] == bench.METRIC
    assert out["value"] > 0 and out["higher_is_better"] is True and out["dtype"] == "f64"
    assert out["cpu_baseline"]["kind"] == "oracle" and out["cpu_baseline"]["value"] == out["value"]
    assert out["e2e"] == {"value": out["value"], "unit": out["unit"], "h2d_bytes_per_step": 0,
                          "d2h_bytes_per_step": 0}
    assert out["config"]["workload"].startswith("tiny drafting round")
    if not loaded_before:                     # the oracle's arm never touched the library
        assert "paper_2609_37029_gb300.lsp" not in sys.modules


def test_prefix_rows_are_the_rows_fold_keeps():
    """The rows the reference arm folds are request 0's share of the same seeded chunks."""
    sys.path.insert(0, ROOT)
    import bench
    from paper_2609_37029_gb300 import synth
    s = synth.SHAPES["tiny"]
    wl = bench.Workload(s, None, 123, device="cpu")
    rows = wl.prefix_rows(0, bench.FOLD_CHUNK + 5)
    assert [r[0].shape[2] for r in rows] == [bench.FOLD_CHUNK, 5]
    k, v, _ = synth.make_features(s, bench.FOLD_CHUNK, seed=123 + 1, device="cpu", with_h=False)
    assert (rows[1][0] == k[0:1, :, :5]).all() and (rows[1][1] == v[0:1, :, :5]).all()
    _, _, h = synth.make_features(s, bench.FOLD_CHUNK, seed=123 + 7000, device="cpu")
    assert (rows[1][2] == h[0:1, :, 4:5]).all()
