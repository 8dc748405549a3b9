"""tb_decode_workspace_prepare + tb_decode_attn_prepared: the decode step on a
workspace kept from step to step (no per-call clearing kernel).

Checked through the C ABI against tb_decode_attn on the same inputs, over
consecutive calls on one prepared workspace whose lengths change from call to
call: the outputs must be bit-identical (same kernels, same summation order),
which also shows that every call left the split counters at zero for the next
one (a counter left at a non-zero value would keep the next call's last
split CTA from recognising itself, and its output would not be written).
The status word is sticky on this path: a flag stays until the workspace is
prepared again.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import timebill_oracle as orc  # noqa: E402
from paper_2512_21859_gb300 import binding as tb  # noqa: E402
from paper_2512_21859_gb300 import inputs  # noqa: E402
from tests.gpu_common import DT, to_dev  # noqa: E402

pytestmark = pytest.mark.gpu
TOL_OUT = {"f32": 1e-5, "bf16": 2e-2}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2512_21859_gb300 import build
    build.build()
    tb.load()


def _cache(seed, dtype, hq, hkv, d, caps):
    rng = np.random.default_rng(seed)
    offs = np.concatenate([[0], np.cumsum(caps)[:-1]]).astype(np.int64)
    rows = int(np.sum(caps))
    scale = 1 / np.sqrt(d) if dtype == "bf16" else 1.0
    Kc = (rng.standard_normal((hkv, rows, d)) * scale).astype(np.float32)
    Vc = (rng.standard_normal((hkv, rows, d)) * scale).astype(np.float32)
    q = rng.standard_normal((len(caps), hq, d)).astype(np.float32)
    if dtype == "bf16":
        Kc, Vc, q = inputs.f32_to_bf16(Kc), inputs.f32_to_bf16(Vc), inputs.f32_to_bf16(q)
    return offs, rows, q, Kc, Vc


@pytest.mark.parametrize("dtype,hq,hkv,d", [("bf16", 28, 4, 128), ("bf16", 32, 8, 128),
                                            ("bf16", 8, 1, 64), ("f32", 4, 2, 64)])
def test_prepared_matches_per_call_clearing_over_consecutive_steps(dtype, hq, hkv, d):
    caps = [6000, 900, 2100]
    offs, rows, q, Kc, Vc = _cache(hq + d, dtype, hq, hkv, d, caps)
    desc = tb.DecodeDesc(hq=hq, hkv=hkv, head_dim=d, dtype=DT[dtype], cache_offset=offs,
                         cache_cap=caps, cache_rows=rows, max_len=max(caps))
    qd, Kd, Vd = to_dev(q, dtype), to_dev(Kc, dtype), to_dev(Vc, dtype)
    nbytes = tb.tb_decode_workspace_size(desc)
    ws_ref = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    # a prepared workspace starts from garbage: prepare must zero what matters
    ws = torch.full((nbytes,), 0xA5, dtype=torch.uint8, device="cuda")
    tb.tb_decode_workspace_prepare(desc, ws)
    shape = (len(caps), hq, d)
    steps = [[5000, 1, 2000], [5001, 0, 2001], [37, 900, 129], [6000, 899, 2100]]
    for lens in steps:
        lens_d = torch.tensor(lens, dtype=torch.int32, device="cuda")
        ref = torch.empty(shape, dtype=torch.float32, device="cuda")
        got = torch.full(shape, float("nan"), dtype=torch.float32, device="cuda")
        tb.tb_decode_attn(desc, qd, Kd, Vd, lens_d, ref, ws_ref)
        tb.tb_decode_attn_prepared(desc, qd, Kd, Vd, lens_d, got, ws)
        torch.cuda.synchronize()
        assert torch.equal(got, ref), lens
    assert tb.tb_read_status(ws) == (tb.TB_OK, 0)
    # and against the oracle, on the last step
    want = orc.decode_batch(inputs.as_f32(q, dtype), inputs.as_f32(Kc, dtype), inputs.as_f32(Vc, dtype),
                            steps[-1], offs)
    assert np.max(np.abs(got.cpu().numpy() - want)) <= TOL_OUT[dtype]


def test_prepared_status_flag_is_sticky_until_prepared_again():
    caps = [300]
    offs, rows, q, Kc, Vc = _cache(5, "bf16", 8, 2, 128, caps)
    desc = tb.DecodeDesc(hq=8, hkv=2, head_dim=128, dtype=tb.TB_BF16, cache_offset=offs,
                         cache_cap=caps, cache_rows=rows, max_len=512)
    qd, Kd, Vd = to_dev(q, "bf16"), to_dev(Kc, "bf16"), to_dev(Vc, "bf16")
    ws = torch.empty(tb.tb_decode_workspace_size(desc), dtype=torch.uint8, device="cuda")
    tb.tb_decode_workspace_prepare(desc, ws)
    out = torch.empty((1, 8, 128), dtype=torch.float32, device="cuda")
    tb.tb_decode_attn_prepared(desc, qd, Kd, Vd, torch.tensor([400], dtype=torch.int32, device="cuda"),
                               out, ws)                      # above the cap: clamped, flagged
    st, raw = tb.tb_read_status(ws)
    assert st == tb.TB_ERR_INVALID_ARG and raw & 2
    want = orc.decode_batch(inputs.as_f32(q, "bf16"), inputs.as_f32(Kc, "bf16"), inputs.as_f32(Vc, "bf16"),
                            [300], offs)
    assert np.max(np.abs(out.cpu().numpy() - want)) <= TOL_OUT["bf16"]
    tb.tb_decode_attn_prepared(desc, qd, Kd, Vd, torch.tensor([300], dtype=torch.int32, device="cuda"),
                               out, ws)                      # a valid call keeps the flag
    assert tb.tb_read_status(ws)[0] == tb.TB_ERR_INVALID_ARG
    assert np.max(np.abs(out.cpu().numpy() - want)) <= TOL_OUT["bf16"]
    tb.tb_decode_workspace_prepare(desc, ws)                 # prepared again: clear
    assert tb.tb_read_status(ws) == (tb.TB_OK, 0)


@pytest.mark.parametrize("dtype,hq,hkv,d", [("bf16", 28, 4, 128), ("bf16", 32, 8, 128), ("bf16", 8, 1, 64)])
def test_early_cache_read_in_a_decode_loop(dtype, hq, hkv, d):
    """TB_DECODE_EARLY_CACHE_READ in the pattern it is for: every step first
    appends its own K/V row at lens[b] - 1 (here with a copy kernel just
    before the call), then runs tb_decode_attn_prepared with the flag, whose
    kernel requests its first tiles before that copy has completed and reads
    the appended row again after it. Bit-identical to tb_decode_attn on the
    same cache at every step; the appended rows land in every position of a
    tile (the lengths walk across tile and split boundaries)."""
    caps = [700, 300, 2100]
    offs, rows, q, Kc, Vc = _cache(hq * 3 + d, dtype, hq, hkv, d, caps)
    rng = np.random.default_rng(d)
    new_k = inputs.f32_to_bf16((rng.standard_normal((80, hkv, len(caps), d)) / np.sqrt(d)).astype(np.float32))
    new_v = inputs.f32_to_bf16((rng.standard_normal((80, hkv, len(caps), d)) / np.sqrt(d)).astype(np.float32))
    qd, Kd, Vd = to_dev(q, dtype), to_dev(Kc, dtype), to_dev(Vc, dtype)
    nk, nv = to_dev(new_k, dtype), to_dev(new_v, dtype)
    start = [600, 1, 1950]
    base = dict(hq=hq, hkv=hkv, head_dim=d, dtype=DT[dtype], cache_offset=offs, cache_cap=caps, cache_rows=rows)
    top = tb.DecodeDesc(max_len=max(caps), flags=tb.TB_DECODE_EARLY_CACHE_READ, **base)
    ws = torch.empty(tb.tb_decode_workspace_size(top), dtype=torch.uint8, device="cuda")
    tb.tb_decode_workspace_prepare(top, ws)
    ws_ref = torch.empty_like(ws)
    shape = (len(caps), hq, d)
    out = torch.empty(shape, dtype=torch.float32, device="cuda")
    ref = torch.empty(shape, dtype=torch.float32, device="cuda")
    for step in range(80):
        lens = [x + step for x in start]
        for b in range(len(caps)):     # the step's own row, appended just before the call
            Kd[:, offs[b] + lens[b] - 1] = nk[step, :, b]
            Vd[:, offs[b] + lens[b] - 1] = nv[step, :, b]
        lens_d = torch.tensor(lens, dtype=torch.int32, device="cuda")
        flagged = tb.DecodeDesc(max_len=max(lens), flags=tb.TB_DECODE_EARLY_CACHE_READ, **base)
        tb.tb_decode_attn_prepared(flagged, qd, Kd, Vd, lens_d, out, ws)
        tb.tb_decode_attn(tb.DecodeDesc(max_len=max(lens), **base), qd, Kd, Vd, lens_d, ref, ws_ref)
        assert torch.equal(out, ref), (step, lens)
    assert tb.tb_read_status(ws) == (tb.TB_OK, 0)
    got = out.cpu().numpy()
    Kf = inputs.as_f32(Kd.view(torch.int16).cpu().numpy().view(np.uint16), dtype)
    Vf = inputs.as_f32(Vd.view(torch.int16).cpu().numpy().view(np.uint16), dtype)
    want = orc.decode_batch(inputs.as_f32(q, dtype), Kf, Vf, lens, offs)
    assert np.max(np.abs(got - want)) <= TOL_OUT[dtype]
