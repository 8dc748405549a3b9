"""Helpers shared by the GPU parity tests: device marshalling through the C
ABI binding, and the acceptance rules for retained index sets."""
import numpy as np

from paper_2512_21859_gb300 import binding as tb
from paper_2512_21859_gb300 import inputs

DT = {"f32": tb.TB_F32, "bf16": tb.TB_BF16}


def to_dev(arr: np.ndarray, dtype: str):
    import torch
    if dtype == "bf16":
        t = torch.from_numpy(np.ascontiguousarray(arr).view(np.int16)).view(torch.bfloat16)
    else:
        t = torch.from_numpy(np.ascontiguousarray(arr, dtype=np.float32))
    return t.cuda()


def from_dev(t, dtype: str) -> np.ndarray:
    import torch
    if dtype == "bf16":
        return t.view(torch.int16).cpu().numpy().view(np.uint16)
    return t.cpu().numpy()


def evict_desc(wl, lay, extra_cap: int = 0, flags: int = 0):
    n, a = lay["n"], lay["alpha"]
    caps = [tb.tb_retained_count_ex(int(nb), wl.window, float(ab), flags)[1] + extra_cap
            for nb, ab in zip(n, a)]
    return tb.EvictDesc(hq=wl.hq, hkv=wl.hkv, head_dim=wl.head_dim, window=wl.window,
                        pool_k=wl.pool_k, dtype=DT[wl.dtype], n=n, alpha=a,
                        kv_offset=lay["kv_offset"], kv_rows=int(np.sum(n)), out_cap=caps, flags=flags)


def run_evict(wl, lay, extra_cap: int = 0, dev=None, flags: int = 0):
    """tb_score_evict on the GPU; returns host copies of idx, pooled, Kc, Vc and the
    device tensors (for decode)."""
    import torch
    desc = evict_desc(wl, lay, extra_cap, flags)
    if dev is None:
        dev = {k: to_dev(lay[k], wl.dtype) for k in ("q_win", "K", "V")}
    score_rows, idx_rows = tb.tb_evict_layout(desc)
    tdt = dev["K"].dtype
    idx = torch.full((wl.hkv, idx_rows), -1, dtype=torch.int32, device="cuda")
    pooled = torch.zeros((wl.hkv, max(score_rows, 1)), dtype=torch.float32, device="cuda")
    Kc = torch.zeros((wl.hkv, desc.out_rows, wl.head_dim), dtype=tdt, device="cuda")
    Vc = torch.zeros_like(Kc)
    ws = torch.empty(tb.tb_evict_workspace_size(desc), dtype=torch.uint8, device="cuda")
    tb.tb_score_evict(desc, dev["q_win"], dev["K"], dev["V"], idx, Kc, Vc, pooled, ws)
    st, raw = tb.tb_read_status(ws)
    assert st == tb.TB_OK, raw
    torch.cuda.synchronize()
    return {"desc": desc, "idx": idx.cpu().numpy(), "pooled": pooled.cpu().numpy(),
            "Kc_t": Kc, "Vc_t": Vc, "ws": ws, "dev": dev}


def request_slices(desc, b):
    """(score column offset, idx column offset) of request b."""
    P = [int(n) - desc.window for n in desc.n]
    R = [tb.tb_retained_count_ex(int(n), desc.window, float(a), desc.flags)[1]
         for n, a in zip(desc.n, desc.alpha)]
    return int(np.sum(P[:b])), int(np.sum(R[:b])), P[b], R[b]


def check_index_set(gpu_idx, oracle_pooled, k, n, window, rel=1e-6):
    """Acceptance rule for one (request, KV head): exactly k prefix positions
    followed by the window, unique and ascending; every position whose oracle
    pooled score lies outside rel * tau of the k-th largest score tau is kept
    or dropped exactly as the oracle decides. Returns the number of excused
    (in-band) positions on which the two sides differ."""
    P = n - window
    gpu_idx = np.asarray(gpu_idx, dtype=np.int64)
    assert gpu_idx.shape[0] == k + window
    assert np.array_equal(gpu_idx[k:], np.arange(P, n))
    pre = gpu_idx[:k]
    assert np.all(np.diff(gpu_idx) > 0)
    assert k == 0 or (pre.min() >= 0 and pre.max() < P)
    if k == 0 or k == P:
        if k == P:
            assert np.array_equal(pre, np.arange(P))
        return 0
    pooled = np.asarray(oracle_pooled, dtype=np.float64)
    tau = np.sort(pooled)[::-1][k - 1]
    band = np.abs(pooled - tau) <= rel * tau
    kept = np.zeros(P, dtype=bool)
    kept[pre] = True
    must_keep = (pooled > tau) & ~band
    must_drop = (pooled < tau) & ~band
    bad_keep = np.nonzero(must_keep & ~kept)[0]
    bad_drop = np.nonzero(must_drop & kept)[0]
    assert bad_keep.size == 0 and bad_drop.size == 0, (
        "outside the 1e-6 band: missing %s, extra %s" % (bad_keep[:10], bad_drop[:10]))
    o_idx = np.lexsort((np.arange(P), -pooled))[:k]
    o_kept = np.zeros(P, dtype=bool)
    o_kept[o_idx] = True
    return int(np.sum(o_kept != kept))
