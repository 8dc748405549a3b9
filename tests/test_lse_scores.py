"""Window scores from given row log-sum-exp values (tb_window_scores_lse).

Oracle pins (no GPU): the normalisers of window_lse against a pure-Python
log-sum-exp with math.fsum, the scores rebuilt from them against the
brute-force voting of tests/brute_force.py, and two properties that hold
for any input: each window row's probabilities over its visible keys sum to
one, and raising every lse by c scales every score by exp(-c).
GPU parity (@gpu): the one-pass kernels against the oracle and against the
two-pass tb_window_scores, for bf16 (tensor-core path) and fp32 (SIMT path).
"""
import math

import numpy as np
import pytest

from oracle import timebill_oracle as orc
from paper_2512_21859_gb300 import inputs
from tests import brute_force as bf


def _tiny(seed, hq=4, hkv=2, W=5, N=23, d=8):
    rng = np.random.default_rng(seed)
    return rng.standard_normal((hq, W, d)), rng.standard_normal((hkv, N, d))


@pytest.mark.parametrize("seed", range(4))
def test_lse_against_pure_python(seed):
    q, K = _tiny(seed)
    hq, W, d = q.shape
    G = hq // K.shape[0]
    P = K.shape[1] - W
    got = orc.window_lse(q, K)
    for h in range(hq):
        for w in range(W):
            logits = [sum(q[h, w, i] * K[h // G, j, i] for i in range(d)) / math.sqrt(d)
                      for j in range(P + w + 1)]
            m = max(logits)
            want = m + math.log(math.fsum(math.exp(x - m) for x in logits))
            assert got[h, w] == pytest.approx(want, abs=1e-12)


@pytest.mark.parametrize("seed", range(4))
def test_scores_from_lse_match_brute_force_voting(seed):
    q, K = _tiny(seed)
    G = q.shape[0] // K.shape[0]
    S = orc.window_scores_from_lse(q, K, orc.window_lse(q, K))
    ref = bf.scores(q.tolist(), K.tolist(), G)
    np.testing.assert_allclose(S, np.array(ref), rtol=1e-12, atol=0)
    # and the two-pass definition
    np.testing.assert_allclose(S, orc.window_scores(q, K), rtol=1e-12, atol=0)


def test_rows_sum_to_one_and_shift_scales():
    q, K = _tiny(11, hq=6, hkv=3, W=7, N=40, d=16)
    hq, W, d = q.shape
    G = hq // K.shape[0]
    P = K.shape[1] - W
    L = orc.window_lse(q, K)
    for h in range(hq):
        for w in range(W):
            s = (q[h, w] @ K[h // G, :P + w + 1].T) / math.sqrt(d)
            assert math.fsum(np.exp(s - L[h, w])) == pytest.approx(1.0, abs=1e-13)
    S0 = orc.window_scores_from_lse(q, K, L)
    S1 = orc.window_scores_from_lse(q, K, L + 0.75)
    np.testing.assert_allclose(S1, S0 * math.exp(-0.75), rtol=1e-13)


# ---------------------------------------------------------------------------
# GPU parity
# ---------------------------------------------------------------------------

def _gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2512_21859_gb300 import binding as tb, build
    build.build()
    tb.load()
    return torch, tb


def _lse_of(wl, lay):
    """fp64 oracle normalisers of every request, packed [B][Hq][W] as fp32."""
    q = inputs.as_f32(lay["q_win"], wl.dtype)
    K = inputs.as_f32(lay["K"], wl.dtype)
    out = []
    for b, n in enumerate(lay["n"]):
        off = int(lay["kv_offset"][b])
        out.append(orc.window_lse(q[b], K[:, off:off + int(n)]))
    return np.stack(out).astype(np.float32)


@pytest.mark.gpu
@pytest.mark.parametrize("dtype,hq,hkv,d,W,ns", [
    ("bf16", 28, 4, 128, 32, [5000, 1200]),   # tensor-core kernel, two requests, ragged tails
    ("bf16", 32, 8, 128, 64, [2100]),         # 256 window rows per KV head
    ("bf16", 8, 2, 64, 16, [777, 300]),       # head_dim 64
    ("f32", 4, 2, 64, 16, [512, 97]),         # SIMT kernel
])
def test_gpu_scores_from_lse_match_oracle(dtype, hq, hkv, d, W, ns):
    torch, tb = _gpu()
    from tests.gpu_common import request_slices, to_dev
    wl = inputs.Workload(name="lse", layers=1, hq=hq, hkv=hkv, head_dim=d, dtype=dtype, batch=len(ns),
                         window=W, pool_k=7, decode_steps=1, seed=31, n_fixed=ns[0], alpha=0.5,
                         heavy_frac=0.01, unit_keys=dtype == "bf16")
    lay = inputs.make_layer(wl, 0, n_override=ns)
    lay["alpha"] = np.full(len(ns), 0.5)
    desc = tb.EvictDesc(hq=hq, hkv=hkv, head_dim=d, window=W, pool_k=7,
                        dtype=tb.TB_BF16 if dtype == "bf16" else tb.TB_F32, n=lay["n"], alpha=lay["alpha"])
    score_rows, _ = tb.tb_evict_layout(desc)
    lse = _lse_of(wl, lay)
    ws = torch.empty(tb.tb_evict_workspace_size(desc), dtype=torch.uint8, device="cuda")
    one = torch.zeros((hkv, score_rows), dtype=torch.float32, device="cuda")
    two = torch.zeros_like(one)
    qd, Kd = to_dev(lay["q_win"], dtype), to_dev(lay["K"], dtype)
    tb.tb_window_scores_lse(desc, qd, Kd, torch.from_numpy(lse).cuda(), one, ws)
    st, raw = tb.tb_read_status(ws)
    assert st == tb.TB_OK, raw
    tb.tb_window_scores(desc, qd, Kd, two, ws)
    got, got2 = one.cpu().numpy(), two.cpu().numpy()
    q = inputs.as_f32(lay["q_win"], dtype)
    K = inputs.as_f32(lay["K"], dtype)
    for b, n in enumerate(ns):
        s0, _, P, _ = request_slices(desc, b)
        off = int(lay["kv_offset"][b])
        # the oracle from the same fp32-rounded normalisers the kernel read
        ref = orc.window_scores_from_lse(q[b], K[:, off:off + n], lse[b].astype(np.float64))
        # (the kernel turns lse into log2 units in fp32: one more rounding of
        # a value near 25, ~1e-6 relative on each exponential at most)
        np.testing.assert_allclose(got[:, s0:s0 + P], ref, rtol=3e-6, atol=0)
        # and the two-pass call, whose normalisers it computes itself
        np.testing.assert_allclose(got[:, s0:s0 + P], got2[:, s0:s0 + P], rtol=4e-6, atol=0)


@pytest.mark.gpu
def test_gpu_lse_rejects_bad_pointers():
    torch, tb = _gpu()
    desc = tb.EvictDesc(hq=4, hkv=2, head_dim=64, window=16, pool_k=7, dtype=tb.TB_F32, n=[64], alpha=[0.5])
    ws = torch.empty(tb.tb_evict_workspace_size(desc), dtype=torch.uint8, device="cuda")
    q = torch.zeros((1, 4, 16, 64), device="cuda")
    K = torch.zeros((2, 64, 64), device="cuda")
    S = torch.zeros((2, 64), device="cuda")
    with pytest.raises(tb.TbError) as e:
        tb.tb_window_scores_lse(desc, q, K, None, S, ws)
    assert e.value.status == tb.TB_ERR_INVALID_ARG


@pytest.mark.gpu
def test_gpu_lse_128k_sampled_heads():
    """The one-pass call at the full 128K size the benchmark times
    (32q/8kv, N 131072, W 64): KV heads 0 and 7 recomputed by the oracle from
    the same fp32 normalisers; the other heads get finite stand-ins."""
    torch, tb = _gpu()
    from tests.gpu_common import to_dev
    wl = inputs.WORKLOADS["128k"]
    lay = inputs.make_layer(wl, 0)
    n = int(lay["n"][0])
    q = inputs.as_f32(lay["q_win"], "bf16")
    K = inputs.as_f32(lay["K"], "bf16")
    G = wl.group
    lse = np.zeros((1, wl.hq, wl.window), dtype=np.float32)
    heads = (0, 7)
    for g in heads:
        lse[0, g * G:(g + 1) * G] = orc.window_lse(q[0, g * G:(g + 1) * G], K[g:g + 1, :n]).astype(np.float32)
    desc = tb.EvictDesc(hq=wl.hq, hkv=wl.hkv, head_dim=wl.head_dim, window=wl.window, pool_k=wl.pool_k,
                        dtype=tb.TB_BF16, n=lay["n"], alpha=lay["alpha"])
    score_rows, _ = tb.tb_evict_layout(desc)
    scores = torch.zeros((wl.hkv, score_rows), dtype=torch.float32, device="cuda")
    ws = torch.empty(tb.tb_evict_workspace_size(desc), dtype=torch.uint8, device="cuda")
    tb.tb_window_scores_lse(desc, to_dev(lay["q_win"], "bf16"), to_dev(lay["K"], "bf16"),
                            torch.from_numpy(lse).cuda(), scores, ws)
    st, raw = tb.tb_read_status(ws)
    assert st == tb.TB_OK, raw
    got = scores.cpu().numpy()
    for g in heads:
        ref = orc.window_scores_from_lse(q[0, g * G:(g + 1) * G], K[g:g + 1, :n],
                                         lse[0, g * G:(g + 1) * G].astype(np.float64))
        np.testing.assert_allclose(got[g], ref[0], rtol=3e-6, atol=0)
