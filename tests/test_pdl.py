"""Programmatic dependent launch keeps stream order: the select -> gather ->
decode chain replayed from a CUDA graph gives bit-identical outputs with PDL
(the default) and with TB_NO_PDL set (ordinary launches)."""
import os
import subprocess
import sys

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))


@pytest.mark.gpu
def test_pdl_chain_matches_ordinary_launches(tmp_path):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2512_21859_gb300 import build
    build.build()
    res = {}
    for name, extra in (("pdl", {}), ("plain", {"TB_NO_PDL": "1"})):
        env = {k: v for k, v in os.environ.items() if k != "TB_NO_PDL"}
        env.update(extra)
        path = str(tmp_path / (name + ".npz"))
        subprocess.run([sys.executable, os.path.join(HERE, "pdl_chain.py"), path], env=env, check=True,
                       timeout=600)
        res[name] = np.load(path)
    for key in ("idx", "Kc", "Vc", "out"):
        assert np.array_equal(res["pdl"][key], res["plain"][key]), key
    assert (res["pdl"]["idx"] >= 0).all()
