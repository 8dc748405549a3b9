"""tb_decode_attn_noalloc: decode attention for callers that cannot allocate.

A serving loop under a hard deadline may forbid allocator calls on its
per-token path, and a plugin inside a host framework may have no allocator
at all; this entry point takes no workspace and uses the library's own
device array instead. These tests call it through the C ABI and check it
against tb_decode_attn (which takes a caller workspace) on the same inputs,
on two calls in a row, so the second call also proves that leftovers of the
first call in the shared array do not leak into its result.

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
                         cache_offset=offs, cache_cap=caps, cache_rows=rows, max_len=max(lens))
    return desc, q, Kc, Vc, lens


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
def test_noalloc_matches_workspace_entry_on_two_calls(lib):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    cases = [
        ("bf16", _case(1, "bf16", 28, 4, 128, [4097, 1, 300, 2080])),   # GQA 7:1, ragged lengths
        ("f32", _case(2, "f32", 4, 2, 64, [272, 0, 33])),               # a zero length in the batch
    ]
    for dtype, (desc, q, Kc, Vc, lens) in cases:
        assert tb.tb_decode_workspace_size(desc) <= tb.TB_NOALLOC_SCRATCH_BYTES
        qd, Kd, Vd = _dev(q, dtype), _dev(Kc, dtype), _dev(Vc, dtype)
        lens_d = torch.tensor(lens, dtype=torch.int32, device="cuda")
        shape = (desc.batch, desc.hq, desc.head_dim)
        ref = torch.empty(shape, dtype=torch.float32, device="cuda")
        ws = torch.empty(tb.tb_decode_workspace_size(desc), dtype=torch.uint8, device="cuda")
        tb.tb_decode_attn(desc, qd, Kd, Vd, lens_d, ref, ws)
        got = torch.full(shape, float("nan"), dtype=torch.float32, device="cuda")
        tb.tb_decode_attn_noalloc(desc, qd, Kd, Vd, lens_d, got)
        torch.cuda.synchronize()
        err = float((got - ref).abs().max().item())
        assert err <= TOL_OUT[dtype], (dtype, err)
        assert not torch.isnan(got).any()
