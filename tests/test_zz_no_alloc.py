"""tb_decode_attn_noalloc: decode attention for callers that cannot allocate.

A serving loop under a hard deadline may forbid allocator calls on its
per-token path (an allocation can synchronise the device and take unbounded
time), and a plugin inside a host framework may have no allocator at all;
this entry point takes no workspace and uses the library's own device array
instead. These tests call it through the C ABI:
  * against tb_decode_attn on the same inputs, bit for bit (the same kernels,
    split layout and summation order, so any leftover of an earlier call in
    the shared array would change bits), and against the CPU oracle within
    the decode tolerances of the parity tests;
  * on one descriptor twice, with other queries and lengths the second time
    and a call of another shape in between, so that the second call also
    shows that the first call's contents in the shared array do not leak;
  * with a length above its cap, whose flag tb_decode_noalloc_status reads
    back (and the next call clears).

This file is named so that pytest collects it last.
"""
import numpy as np
import pytest

from paper_2512_21859_gb300 import binding as tb
from paper_2512_21859_gb300 import inputs

TOL_OUT = {"f32": 1e-5, "bf16": 2e-2}   # the decode tolerances of the parity tests


@pytest.fixture(scope="module")
def lib():
    from paper_2512_21859_gb300 import build
    build.build()
    tb.load()
    return tb


def _case(seed, dtype, hq, hkv, d, lens):
    rng = np.random.default_rng(seed)
    caps = [max(x, 1) + 3 for x in lens]
    offs = np.concatenate([[0], np.cumsum(caps)[:-1]]).astype(np.int64)
    rows = int(np.sum(caps))
    scale = 1 / np.sqrt(d) if dtype == "bf16" else 1.0
    Kc = (rng.standard_normal((hkv, rows, d)) * scale).astype(np.float32)
    Vc = (rng.standard_normal((hkv, rows, d)) * scale).astype(np.float32)
    q = rng.standard_normal((len(lens), hq, d)).astype(np.float32)
    if dtype == "bf16":
        Kc, Vc, q = inputs.f32_to_bf16(Kc), inputs.f32_to_bf16(Vc), inputs.f32_to_bf16(q)
    desc = tb.DecodeDesc(hq=hq, hkv=hkv, head_dim=d, dtype=tb.TB_BF16 if dtype == "bf16" else tb.TB_F32,
                         cache_offset=offs, cache_cap=caps, cache_rows=rows, max_len=max(caps))
    return desc, q, Kc, Vc


def _dev(x, dtype):
    import torch
    if dtype == "bf16":
        return torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).view(torch.bfloat16).cuda()
    return torch.from_numpy(np.ascontiguousarray(x)).cuda()


def test_oversized_descriptor_is_rejected_before_launch(lib):
    # 64 requests x 128 query heads x d 128 of fp32 split partials: beyond 4 MiB
    desc = tb.DecodeDesc(hq=128, hkv=8, head_dim=128, dtype=tb.TB_BF16, cache_offset=np.arange(64) * 100000,
                         cache_cap=[100000] * 64, cache_rows=6400000, max_len=100000)
    assert tb.tb_decode_workspace_size(desc) > tb.TB_NOALLOC_SCRATCH_BYTES
    fake = 1 << 20
    with pytest.raises(tb.TbError) as e:
        tb.tb_decode_attn_noalloc(desc, fake, fake, fake, fake, fake, stream=0)
    assert e.value.status == tb.TB_ERR_WORKSPACE


@pytest.mark.gpu
def test_noalloc_matches_workspace_entry_and_oracle_on_repeated_calls(lib):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from oracle import timebill_oracle as orc

    def run(desc, dtype, q, Kd, Vd, Kc, Vc, lens):
        """One no-allocation call against tb_decode_attn (own workspace) and
        the oracle on the same inputs; returns the output."""
        assert tb.tb_decode_workspace_size(desc) <= tb.TB_NOALLOC_SCRATCH_BYTES
        qd = _dev(q, dtype)
        lens_d = torch.tensor(lens, dtype=torch.int32, device="cuda")
        shape = (desc.batch, desc.hq, desc.head_dim)
        ref = torch.empty(shape, dtype=torch.float32, device="cuda")
        ws = torch.empty(tb.tb_decode_workspace_size(desc), dtype=torch.uint8, device="cuda")
        tb.tb_decode_attn(desc, qd, Kd, Vd, lens_d, ref, ws)
        got = torch.full(shape, float("nan"), dtype=torch.float32, device="cuda")
        tb.tb_decode_attn_noalloc(desc, qd, Kd, Vd, lens_d, got)
        assert tb.tb_decode_noalloc_status() == (tb.TB_OK, 0)
        assert tb.tb_read_status(ws) == (tb.TB_OK, 0)
        assert torch.equal(got, ref), dtype
        want = orc.decode_batch(inputs.as_f32(q, dtype), inputs.as_f32(Kc, dtype), inputs.as_f32(Vc, dtype),
                                lens, desc.cache_offset)
        err = float(np.max(np.abs(got.cpu().numpy() - want)))
        assert err <= TOL_OUT[dtype], (dtype, err)
        return got

    # A: GQA 7:1, ragged lengths; B: fp32 with a zero length in the batch
    dA, qA, KA, VA = _case(1, "bf16", 28, 4, 128, [4097, 1, 300, 2080])
    dB, qB, KB, VB = _case(2, "f32", 4, 2, 64, [272, 0, 33])
    KAd, VAd = _dev(KA, "bf16"), _dev(VA, "bf16")
    KBd, VBd = _dev(KB, "f32"), _dev(VB, "f32")
    first = run(dA, "bf16", qA, KAd, VAd, KA, VA, [4097, 1, 300, 2080])
    run(dB, "f32", qB, KBd, VBd, KB, VB, [272, 0, 33])
    # A again: other queries and lengths on the same descriptor
    qA2 = inputs.f32_to_bf16(np.random.default_rng(7).standard_normal(qA.shape).astype(np.float32))
    second = run(dA, "bf16", qA2, KAd, VAd, KA, VA, [3000, 4, 299, 2079])
    assert not torch.equal(first, second)


@pytest.mark.gpu
def test_noalloc_length_flag_reads_back(lib):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    desc, q, Kc, Vc = _case(3, "bf16", 8, 2, 128, [300])     # cap 303
    qd, Kd, Vd = _dev(q, "bf16"), _dev(Kc, "bf16"), _dev(Vc, "bf16")
    out = torch.empty((1, 8, 128), dtype=torch.float32, device="cuda")
    tb.tb_decode_attn_noalloc(desc, qd, Kd, Vd, torch.tensor([400], dtype=torch.int32, device="cuda"), out)
    st, raw = tb.tb_decode_noalloc_status()
    assert st == tb.TB_ERR_INVALID_ARG and raw & 2
    tb.tb_decode_attn_noalloc(desc, qd, Kd, Vd, torch.tensor([303], dtype=torch.int32, device="cuda"), out)
    assert tb.tb_decode_noalloc_status() == (tb.TB_OK, 0)
