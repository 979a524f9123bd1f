"""C ABI checks that need no GPU: the library loads, exports every entry point
include/lsp.h declares, validates configs on the host, and sizes the state
exactly as the paper's fixed-size interface (Sec. 2.4 "Fixed-cost complexity")."""
import os
import re
import subprocess
import sys

import pytest

import oracle
from paper_2609_37029_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "lsp.h")


@pytest.fixture(scope="module")
def lsp():
    from paper_2609_37029_gb300 import build
    build.build()
    from paper_2609_37029_gb300 import lsp as mod
    return mod


def _declared():
    txt = open(HEADER).read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return sorted(set(re.findall(r"\b(lsp_[a-z_0-9]+)\s*\(", txt)))


def test_every_declared_symbol_is_exported(lsp):
    names = _declared()
    assert "lsp_view_update" in names and "lsp_draft" in names and "lsp_sample" in names
    out = subprocess.run(["nm", "-D", "--defined-only", lsp.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT\s+(lsp_\w+)", out))
    missing = [n for n in names if n not in exported]
    assert not missing, missing
    assert set(lsp.EXPORTED) == set(names)


@pytest.mark.parametrize("name", list(synth.SHAPES))
def test_workload_configs_are_supported(lsp, name):
    cfg = lsp.make_config(synth.SHAPES[name])
    assert lsp.lsp_config_check(cfg) == lsp.LSP_OK


@pytest.mark.parametrize("name", list(synth.SHAPES))
def test_state_bytes_is_the_closed_form(lsp, name):
    s = synth.SHAPES[name]
    es = 2 if s.dtype == "bf16" else 4
    want = s.C * (oracle.state_bytes_per_request(s, elem_bytes=es) + 8)   # + int64 t per request
    assert lsp.lsp_state_bytes(lsp.make_config(s)) == want


def test_state_bytes_at_qwen3_8b_shape_is_6p3_mib_per_request(lsp):
    s = synth.Q8B
    per = lsp.lsp_state_bytes(lsp.make_config(s)) / s.C
    assert abs(per / 2 ** 20 - 6.3) < 0.05


@pytest.mark.parametrize("field,value", [("nq", 7), ("d", 96), ("B", 17), ("V", 1000), ("rc", 40),
                                         ("C", 65), ("H", 200), ("F", 100)])
def test_unsupported_shapes_are_rejected_on_the_host(lsp, field, value):
    cfg = lsp.make_config(synth.Q8B)
    setattr(cfg, field, value)
    assert lsp.lsp_config_check(cfg) == lsp.LSP_ERR_SHAPE
    assert lsp.lsp_state_bytes(cfg) == 0


def test_bad_layer_map_and_null_args(lsp):
    cfg = lsp.make_config(synth.SMALL)
    cfg.layer_map[1] = 4                      # only 4 tapped layers
    assert lsp.lsp_config_check(cfg) == lsp.LSP_ERR_SHAPE
    assert lsp._f["lsp_config_check"](None) == lsp.LSP_ERR_ARG
    assert lsp._f["lsp_draft"](None, None, None, None, None, None, None) == lsp.LSP_ERR_ARG
    assert lsp._f["lsp_view_update"](None, None, None, None) == lsp.LSP_ERR_ARG
    assert lsp.lsp_status_string(lsp.LSP_ERR_TIMEOUT) == "device wait timed out"


def test_the_binding_refuses_to_run_without_its_library(tmp_path):
    """No fallback: a copy of the package without liblsp.so fails at import, loudly."""
    pkg = tmp_path / "paper_2609_37029_gb300"
    pkg.mkdir()
    for name in ("__init__.py", "lsp.py", "synth.py"):
        (pkg / name).write_text(open(os.path.join(ROOT, "paper_2609_37029_gb300", name)).read())
    r = subprocess.run([sys.executable, "-c", "import paper_2609_37029_gb300.lsp"], cwd=tmp_path,
                       capture_output=True, text=True, env={**os.environ, "PYTHONPATH": str(tmp_path)})
    assert r.returncode != 0
    assert "ImportError" in r.stderr and "liblsp.so" in r.stderr


def test_ablation_configs_on_the_host(lsp):
    """W = 0, R = 0 and LSP_NO_BOUNDARY are valid configs whose interface drops exactly the
    removed source's bytes; unknown flag bits are rejected."""
    s = synth.Q8B
    full = lsp.lsp_state_bytes(lsp.make_config(s))
    for variant in ({"W": 0}, {"R": 0}, {"no_boundary": True}):
        v = s.with_(**variant)
        cfg = lsp.make_config(v)
        assert lsp.lsp_config_check(cfg) == lsp.LSP_OK
        assert lsp.lsp_state_bytes(cfg) == s.C * oracle.state_bytes_per_request(v) + 8 * s.C
    assert lsp.lsp_state_bytes(lsp.make_config(s.with_(no_boundary=True))) == full - s.C * s.L * s.H * 2
    cfg = lsp.make_config(s)
    cfg.flags = 2
    assert lsp.lsp_config_check(cfg) == lsp.LSP_ERR_ARG
