"""Failure detection: the bounded device-side waits behind TB_ERR_TIMEOUT.

Every kernel of the library waits on its barriers with a time limit and, when
it runs out, raises the workspace status word, waits for its own copies in
flight, frees its tensor memory and returns, so that the context stays
usable and tb_read_status reports TB_ERR_TIMEOUT. A real kernel only waits
that long when something is broken, so tb_diag_bounded_wait runs the same
exit on purpose with nothing broken: it waits on a barrier that nothing
completes, with a short limit. No GPU is faulted, trapped or hung: the wait
ends by itself after the limit.
"""
import time

import numpy as np
import pytest

from paper_2512_21859_gb300 import binding as tb
from paper_2512_21859_gb300 import inputs


@pytest.fixture(scope="module")
def lib():
    from paper_2512_21859_gb300 import build
    build.build()
    tb.load()
    return tb


@pytest.mark.parametrize("nbytes,limit,arrive,status", [
    (256 + 4096, 5_000, 0, tb.TB_ERR_INVALID_ARG),          # limit below 10 us
    (256 + 4096, 2_000_000_000, 0, tb.TB_ERR_INVALID_ARG),  # limit above 1 s
    (256 + 4096, 100_000, 2, tb.TB_ERR_INVALID_ARG),        # arrive not 0 / 1
    (256 + 4095, 100_000, 0, tb.TB_ERR_WORKSPACE),          # workspace too small
])
def test_wait_diagnostic_rejects_before_launch(lib, nbytes, limit, arrive, status):
    fake = 1 << 20   # never dereferenced: the arguments fail first
    with pytest.raises(tb.TbError) as e:
        tb.tb_diag_bounded_wait(fake, limit, arrive, workspace_bytes=nbytes, stream=0)
    assert e.value.status == status


def test_wait_diagnostic_rejects_misaligned_workspace(lib):
    with pytest.raises(tb.TbError) as e:
        tb.tb_diag_bounded_wait((1 << 20) + 16, 100_000, 0, workspace_bytes=8192, stream=0)
    assert e.value.status == tb.TB_ERR_WORKSPACE


@pytest.mark.gpu
def test_bounded_wait_times_out_and_context_stays_usable(lib):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from oracle import timebill_oracle as orc
    ws = torch.zeros(8192, dtype=torch.uint8, device="cuda")
    # a barrier nothing completes, 200 us limit: the kernel gives up and returns
    t0 = time.perf_counter()
    tb.tb_diag_bounded_wait(ws, 200_000, arrive=0)
    st, raw = tb.tb_read_status(ws)
    assert time.perf_counter() - t0 < 5.0
    assert st == tb.TB_ERR_TIMEOUT and raw & 1, (st, raw)
    # the same exit path with the barrier completed: no flag
    tb.tb_diag_bounded_wait(ws, 200_000, arrive=1)
    assert tb.tb_read_status(ws) == (tb.TB_OK, 0)
    # the context still works: a decode step on the same stream after a timeout
    tb.tb_diag_bounded_wait(ws, 50_000, arrive=0)
    rng = np.random.default_rng(3)
    hq, hkv, d, n = 8, 2, 128, 1000
    Kc = inputs.f32_to_bf16((rng.standard_normal((hkv, n, d)) / np.sqrt(d)).astype(np.float32))
    Vc = inputs.f32_to_bf16((rng.standard_normal((hkv, n, d)) / np.sqrt(d)).astype(np.float32))
    q = inputs.f32_to_bf16(rng.standard_normal((1, hq, d)).astype(np.float32))

    def dev(x):
        return torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).view(torch.bfloat16).cuda()

    desc = tb.DecodeDesc(hq=hq, hkv=hkv, head_dim=d, dtype=tb.TB_BF16, cache_offset=[0], cache_cap=[n],
                         cache_rows=n, max_len=n)
    dws = torch.empty(tb.tb_decode_workspace_size(desc), dtype=torch.uint8, device="cuda")
    out = torch.empty((1, hq, d), dtype=torch.float32, device="cuda")
    tb.tb_decode_attn(desc, dev(q), dev(Kc), dev(Vc), torch.tensor([n], dtype=torch.int32, device="cuda"),
                      out, dws)
    assert tb.tb_read_status(dws) == (tb.TB_OK, 0)
    assert tb.tb_read_status(ws)[0] == tb.TB_ERR_TIMEOUT
    want = orc.decode_batch(inputs.as_f32(q, "bf16"), inputs.as_f32(Kc, "bf16"), inputs.as_f32(Vc, "bf16"),
                            [n], [0])
    assert np.max(np.abs(out.cpu().numpy() - want)) <= 2e-2
