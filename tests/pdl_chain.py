"""Runs select -> gather -> decode, captured in one CUDA graph and replayed
three times, and saves every output to the .npz named on the command line.
tests/test_pdl.py runs it with and without TB_NO_PDL (the switch is read once
per process) and compares the two."""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2512_21859_gb300 import binding as tb  # noqa: E402


def main(path):
    tb.load()
    rng = np.random.default_rng(21)
    hq, hkv, d, W = 32, 8, 128, 64
    ns = [9000, 3001]
    alphas = [0.8, 0.5]
    desc = tb.EvictDesc(hq=hq, hkv=hkv, head_dim=d, window=W, pool_k=7, dtype=tb.TB_BF16, n=ns,
                        alpha=alphas, out_cap=[tb.tb_retained_count(n, W, a)[1] + 1 for n, a in zip(ns, alphas)])
    score_rows, idx_rows = tb.tb_evict_layout(desc)
    S = torch.from_numpy((rng.exponential(1.0, (hkv, score_rows)) ** 3).astype(np.float32)).cuda()
    K = torch.from_numpy(rng.standard_normal((hkv, sum(ns), d), dtype=np.float32) * 0.09).cuda().to(torch.bfloat16)
    V = torch.from_numpy(rng.standard_normal((hkv, sum(ns), d), dtype=np.float32) * 0.09).cuda().to(torch.bfloat16)
    Kc = torch.zeros((hkv, desc.out_rows, d), dtype=torch.bfloat16, device="cuda")
    Vc = torch.zeros_like(Kc)
    idx = torch.full((hkv, idx_rows), -1, dtype=torch.int32, device="cuda")
    ews = torch.empty(tb.tb_evict_workspace_size(desc), dtype=torch.uint8, device="cuda")
    R = [tb.tb_retained_count(n, W, a)[1] for n, a in zip(ns, alphas)]
    ddesc = tb.DecodeDesc(hq=hq, hkv=hkv, head_dim=d, dtype=tb.TB_BF16, cache_offset=desc.out_offset,
                          cache_cap=desc.out_cap, cache_rows=desc.out_rows, max_len=max(R))
    dws = torch.empty(tb.tb_decode_workspace_size(ddesc), dtype=torch.uint8, device="cuda")
    q = torch.from_numpy(rng.standard_normal((len(ns), hq, d), dtype=np.float32)).cuda().to(torch.bfloat16)
    lens = torch.tensor(R, dtype=torch.int32, device="cuda")
    out = torch.empty((len(ns), hq, d), dtype=torch.float32, device="cuda")
    cap = torch.cuda.Stream()

    def chain(st):
        tb.tb_select_topk(desc, S, idx, None, ews, stream=st)
        tb.tb_gather_kv(desc, idx, K, V, Kc, Vc, stream=st)
        tb.tb_decode_attn(ddesc, q, Kc, Vc, lens, out, dws, stream=st)

    chain(torch.cuda.current_stream())
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=cap):
        chain(cap)
    for _ in range(3):
        Kc.zero_()
        Vc.zero_()
        out.zero_()
        g.replay()
    torch.cuda.synchronize()
    assert tb.tb_read_status(dws)[0] == tb.TB_OK
    np.savez(path, idx=idx.cpu().numpy(), Kc=Kc.view(torch.int16).cpu().numpy(),
             Vc=Vc.view(torch.int16).cpu().numpy(), out=out.cpu().numpy())


if __name__ == "__main__":
    main(sys.argv[1])
