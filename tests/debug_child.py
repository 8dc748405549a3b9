"""Child process of tests/test_debug_build.py: runs one eviction and one
decode step of a 7B-shaped bf16 layer through whichever library TB_LIBRARY
selects, then the eviction again with one non-finite window query element,
and writes the outputs and status words to the .npz path given as argv[1]."""
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2512_21859_gb300 import binding as tb  # noqa: E402
from paper_2512_21859_gb300 import inputs  # noqa: E402
from tests.gpu_common import evict_desc, run_evict, to_dev  # noqa: E402


def evict_status(wl, lay):
    """tb_score_evict on the layer, returning the workspace status word."""
    desc = evict_desc(wl, lay)
    dev = {k: to_dev(lay[k], wl.dtype) for k in ("q_win", "K", "V")}
    score_rows, idx_rows = tb.tb_evict_layout(desc)
    idx = torch.empty((wl.hkv, idx_rows), dtype=torch.int32, device="cuda")
    Kc = torch.zeros((wl.hkv, desc.out_rows, wl.head_dim), dtype=dev["K"].dtype, device="cuda")
    Vc = torch.zeros_like(Kc)
    ws = torch.empty(tb.tb_evict_workspace_size(desc), dtype=torch.uint8, device="cuda")
    tb.tb_score_evict(desc, dev["q_win"], dev["K"], dev["V"], idx, Kc, Vc, None, ws)
    return tb.tb_read_status(ws)


def main(path):
    tb.load()
    wl = inputs.WORKLOADS["7b"]
    lay = inputs.make_layer(wl, 0)
    lay = dict(lay, alpha=np.array([0.5]))
    res = run_evict(wl, lay, extra_cap=1)
    st, raw = tb.tb_read_status(res["ws"])
    desc = res["desc"]
    R = int(desc.out_cap[0]) - 1
    step = inputs.make_decode_step(wl, 0, 1, 1)
    Kc, Vc = res["Kc_t"], res["Vc_t"]
    Kc[:, R] = to_dev(step["k_new"][:, 0], wl.dtype)
    Vc[:, R] = to_dev(step["v_new"][:, 0], wl.dtype)
    dd = tb.DecodeDesc(hq=wl.hq, hkv=wl.hkv, head_dim=wl.head_dim, dtype=tb.TB_BF16,
                       cache_offset=desc.out_offset, cache_cap=desc.out_cap,
                       cache_rows=desc.out_rows, max_len=R + 1)
    dws = torch.empty(tb.tb_decode_workspace_size(dd), dtype=torch.uint8, device="cuda")
    out = torch.empty((1, wl.hq, wl.head_dim), dtype=torch.float32, device="cuda")
    lens = torch.tensor([R + 1], dtype=torch.int32, device="cuda")
    tb.tb_decode_attn(dd, to_dev(step["q"], wl.dtype), Kc, Vc, lens, out, dws)
    dst, draw = tb.tb_read_status(dws)
    # one window query element made non-finite: its row's log-sum-exp is NaN
    q_bad = lay["q_win"].copy()
    q_bad.reshape(-1)[0] = np.uint16(0x7FC0)  # bf16 quiet NaN
    bst, braw = evict_status(wl, dict(lay, q_win=q_bad))
    np.savez(path, idx=res["idx"], pooled=res["pooled"], out=out.cpu().numpy(),
             Kc=Kc.view(torch.int16).cpu().numpy())
    print(json.dumps({"library": os.path.basename(tb.library_path()), "evict": [st, raw],
                      "decode": [dst, draw], "nan_query": [bst, braw], "R": R}))


if __name__ == "__main__":
    main(sys.argv[1])
