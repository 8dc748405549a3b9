"""The TB_DEBUG build of the library (libtimebill_kv_debug.so, selected by
TB_LIBRARY=debug): it builds, exports every entry point the header declares,
and on the GPU gives oracle-correct results with a clean status word, while
its device-side checks flag what the release build lets through: a window
query element that is not finite (its row's log-sum-exp is then NaN)."""
import ctypes
import json
import os
import re
import subprocess
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "timebill_kv.h")


def _declared_functions():
    text = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    return sorted(set(re.findall(r"\b(tb_[a-z0-9_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def debug_lib():
    from paper_2512_21859_gb300 import build
    return build.build(debug=True)


def test_debug_library_exports_every_declared_symbol(debug_lib):
    lib = ctypes.CDLL(debug_lib)
    missing = [n for n in _declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_library_path_follows_tb_library(monkeypatch):
    from paper_2512_21859_gb300 import binding
    monkeypatch.setenv("TB_LIBRARY", "debug")
    assert binding.library_path().endswith("libtimebill_kv_debug.so")
    monkeypatch.delenv("TB_LIBRARY")
    assert binding.library_path().endswith("libtimebill_kv.so")


def _run_child(tmp_path, which):
    path = str(tmp_path / ("%s.npz" % which))
    env = dict(os.environ)
    env.pop("TB_LIBRARY", None)
    if which == "debug":
        env["TB_LIBRARY"] = "debug"
    p = subprocess.run([sys.executable, os.path.join(ROOT, "tests", "debug_child.py"), path],
                       capture_output=True, text=True, env=env, cwd=ROOT, timeout=600)
    assert p.returncode == 0, p.stdout[-2000:] + p.stderr[-2000:]
    return json.loads(p.stdout.strip().splitlines()[-1]), np.load(path)


@pytest.mark.gpu
def test_debug_build_on_gpu(debug_lib, tmp_path):
    pytest.importorskip("torch")
    from oracle import timebill_oracle as orc
    from paper_2512_21859_gb300 import binding as tb
    from paper_2512_21859_gb300 import build, inputs
    from tests.gpu_common import check_index_set
    build.build()
    rel, rel_out = _run_child(tmp_path, "release")
    dbg, dbg_out = _run_child(tmp_path, "debug")
    assert rel["library"] == "libtimebill_kv.so" and dbg["library"] == "libtimebill_kv_debug.so"
    # clean inputs: no check fires
    for run in (rel, dbg):
        assert run["evict"][0] == tb.TB_OK and run["decode"][0] == tb.TB_OK, run
    # the planted NaN: only the debug build's normaliser check raises the range bit
    assert rel["nan_query"][0] == tb.TB_OK, rel
    assert dbg["nan_query"][0] == tb.TB_ERR_INVALID_ARG and dbg["nan_query"][1] & 2, dbg
    # the debug build computes what the release build and the oracle do
    wl = inputs.WORKLOADS["7b"]
    lay = inputs.make_layer(wl, 0)
    f = lambda x: inputs.as_f32(x, wl.dtype)  # noqa: E731
    ref = orc.score_evict(f(lay["q_win"]), f(lay["K"]), f(lay["V"]), lay["n"], np.array([0.5]),
                          lay["kv_offset"], wl.window, wl.pool_k)[0]
    n = int(lay["n"][0])
    R = dbg["R"]
    for g in range(wl.hkv):
        check_index_set(dbg_out["idx"][g, :R], ref["pooled"][g], ref["k"], n, wl.window)
        np.testing.assert_allclose(dbg_out["pooled"][g, :n - wl.window], ref["pooled"][g],
                                   rtol=2e-6, atol=0)
    np.testing.assert_allclose(dbg_out["out"], rel_out["out"], rtol=0, atol=2e-2)
