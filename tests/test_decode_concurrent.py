"""The decode's CTA budget (tb_decode_desc.max_ctas), TB_DECODE_CONCURRENT and
TB_EVICT_GATHER_CONCURRENT: a decode step, and the gather of one layer, that
run beside the select of another layer's eviction.

Checked through the C ABI:
- with a CTA budget the keys split fewer ways; the output still matches the
  oracle (decode attention, Eq. 8's N_kv keys), and the prepared path is
  bit-identical to tb_decode_attn for the same descriptor;
- in the schedule the flag is for (window scores, select, then the decode as
  the select's programmatic dependent, sized to the SMs the select leaves
  free, with the gather ordered after the select by an event on a second
  stream), eagerly and replayed from a CUDA graph: the eviction's indices
  and compacted cache are bit-identical to the serial schedule's, the decode
  output is bit-identical to the same descriptor's serial call and matches
  the oracle, and every status word stays clean;
- in the pipelined step (layer B's scores and select, with the decode and
  layer A's gather beside B's select), the same bit-identity with
  tb_score_evict per layer, which itself ignores the gather flag.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import timebill_oracle as orc  # noqa: E402
from paper_2512_21859_gb300 import binding as tb  # noqa: E402
from paper_2512_21859_gb300 import inputs  # noqa: E402
from tests.gpu_common import DT, evict_desc, to_dev  # noqa: E402

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
@pytest.mark.parametrize("max_ctas", [1, 7, 40, 88])
def test_cta_budget_against_oracle(dtype, hq, hkv, d, max_ctas):
    caps = [6000, 900, 2100]
    lens = [5000, 1, 2000]
    offs, rows, q, Kc, Vc = _cache(hq + d + max_ctas, dtype, hq, hkv, d, caps)
    desc = tb.DecodeDesc(hq=hq, hkv=hkv, head_dim=d, dtype=DT[dtype], cache_offset=offs,
                         cache_cap=caps, cache_rows=rows, max_len=max(caps), max_ctas=max_ctas)
    qd, Kd, Vd = to_dev(q, dtype), to_dev(Kc, dtype), to_dev(Vc, dtype)
    nbytes = tb.tb_decode_workspace_size(desc)
    ws_ref = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    ws = torch.full((nbytes,), 0xA5, dtype=torch.uint8, device="cuda")
    tb.tb_decode_workspace_prepare(desc, ws)
    lens_d = torch.tensor(lens, dtype=torch.int32, device="cuda")
    shape = (len(caps), hq, d)
    ref = torch.empty(shape, dtype=torch.float32, device="cuda")
    got = torch.full(shape, float("nan"), dtype=torch.float32, device="cuda")
    tb.tb_decode_attn(desc, qd, Kd, Vd, lens_d, ref, ws_ref)
    tb.tb_decode_attn_prepared(desc, qd, Kd, Vd, lens_d, got, ws)
    torch.cuda.synchronize()
    assert torch.equal(got, ref)
    assert tb.tb_read_status(ws) == (tb.TB_OK, 0)
    assert tb.tb_read_status(ws_ref) == (tb.TB_OK, 0)
    want = orc.decode_batch(inputs.as_f32(q, dtype), inputs.as_f32(Kc, dtype), inputs.as_f32(Vc, dtype),
                            lens, offs)
    assert np.max(np.abs(got.cpu().numpy() - want)) <= TOL_OUT[dtype]


def test_concurrent_flag_has_no_effect_with_the_clearing_kernel():
    caps = [3000, 500]
    offs, rows, q, Kc, Vc = _cache(11, "bf16", 28, 4, 128, caps)
    base = dict(hq=28, hkv=4, head_dim=128, dtype=tb.TB_BF16, cache_offset=offs, cache_cap=caps,
                cache_rows=rows, max_len=max(caps), max_ctas=40)
    qd, Kd, Vd = to_dev(q, "bf16"), to_dev(Kc, "bf16"), to_dev(Vc, "bf16")
    lens_d = torch.tensor([2999, 17], dtype=torch.int32, device="cuda")
    outs = []
    for flags in (0, tb.TB_DECODE_CONCURRENT):
        desc = tb.DecodeDesc(flags=flags, **base)
        ws = torch.empty(tb.tb_decode_workspace_size(desc), dtype=torch.uint8, device="cuda")
        out = torch.empty((2, 28, 128), dtype=torch.float32, device="cuda")
        tb.tb_decode_attn(desc, qd, Kd, Vd, lens_d, out, ws)
        assert tb.tb_read_status(ws) == (tb.TB_OK, 0)
        outs.append(out)
    assert torch.equal(outs[0], outs[1])


def _eviction_buffers(wl, lay, desc):
    score_rows, idx_rows = tb.tb_evict_layout(desc)
    dev = {k: to_dev(lay[k], wl.dtype) for k in ("q_win", "K", "V")}
    out = {"scores": torch.empty((wl.hkv, score_rows), dtype=torch.float32, device="cuda"),
           "idx": torch.full((wl.hkv, idx_rows), -1, dtype=torch.int32, device="cuda"),
           "Kc": torch.zeros((wl.hkv, desc.out_rows, wl.head_dim), dtype=dev["K"].dtype, device="cuda"),
           "ws": torch.empty(tb.tb_evict_workspace_size(desc), dtype=torch.uint8, device="cuda")}
    out["Vc"] = torch.zeros_like(out["Kc"])
    out.update(dev)
    return out


@pytest.mark.parametrize("wl_name,n,alpha", [("7b", 16384, 0.5), ("128k", 40000, 0.9)])
@pytest.mark.parametrize("graph", [False, True])
def test_decode_beside_the_select(wl_name, n, alpha, graph):
    wl = inputs.WORKLOADS[wl_name]
    lay = inputs.make_layer(wl, 3, alpha=alpha, n_override=[n])
    desc = evict_desc(wl, lay)
    # the decode attends over another layer's compacted cache, as in a step
    # that evicts one layer while it decodes the previous one
    caps = [int(desc.out_cap[0]) + 64]
    offs, rows, q, Kc, Vc = _cache(7, "bf16", wl.hq, wl.hkv, wl.head_dim, caps)
    lens = [caps[0] - 5]
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    free = sms - tb.tb_select_ctas(desc)
    assert free > 0
    ddesc = tb.DecodeDesc(hq=wl.hq, hkv=wl.hkv, head_dim=wl.head_dim, dtype=tb.TB_BF16,
                          cache_offset=offs, cache_cap=caps, cache_rows=rows, max_len=caps[0],
                          flags=tb.TB_DECODE_EARLY_CACHE_READ | tb.TB_DECODE_CONCURRENT, max_ctas=free)
    qd, Kd, Vd = to_dev(q, "bf16"), to_dev(Kc, "bf16"), to_dev(Vc, "bf16")
    lens_d = torch.tensor(lens, dtype=torch.int32, device="cuda")
    dws = torch.empty(tb.tb_decode_workspace_size(ddesc), dtype=torch.uint8, device="cuda")
    tb.tb_decode_workspace_prepare(ddesc, dws)

    # serial reference: eviction stages, then the decode on its own
    ser = _eviction_buffers(wl, lay, desc)
    tb.tb_window_scores(desc, ser["q_win"], ser["K"], ser["scores"], ser["ws"])
    tb.tb_select_topk(desc, ser["scores"], ser["idx"], None, ser["ws"])
    tb.tb_gather_kv(desc, ser["idx"], ser["K"], ser["V"], ser["Kc"], ser["Vc"])
    ref_out = torch.empty((1, wl.hq, wl.head_dim), dtype=torch.float32, device="cuda")
    tb.tb_decode_attn_prepared(ddesc, qd, Kd, Vd, lens_d, ref_out, dws)
    torch.cuda.synchronize()
    assert tb.tb_read_status(ser["ws"]) == (tb.TB_OK, 0)

    # the concurrent schedule
    con = _eviction_buffers(wl, lay, desc)
    out = torch.full((1, wl.hq, wl.head_dim), float("nan"), dtype=torch.float32, device="cuda")
    main, side = torch.cuda.Stream(), torch.cuda.Stream()

    def schedule():
        tb.tb_window_scores(desc, con["q_win"], con["K"], con["scores"], con["ws"], stream=main)
        tb.tb_select_topk(desc, con["scores"], con["idx"], None, con["ws"], stream=main)
        side.wait_stream(main)        # the gather after the select's completion
        tb.tb_decode_attn_prepared(ddesc, qd, Kd, Vd, lens_d, out, dws, stream=main)
        tb.tb_gather_kv(desc, con["idx"], con["K"], con["V"], con["Kc"], con["Vc"], stream=side)
        main.wait_stream(side)

    torch.cuda.synchronize()
    if graph:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=main):
            schedule()
        for _ in range(3):
            with torch.cuda.stream(main):
                g.replay()
    else:
        for _ in range(3):
            schedule()
    torch.cuda.synchronize()
    assert tb.tb_read_status(con["ws"]) == (tb.TB_OK, 0)
    assert tb.tb_read_status(dws) == (tb.TB_OK, 0)
    assert torch.equal(con["idx"], ser["idx"])
    assert torch.equal(con["Kc"].view(torch.int16), ser["Kc"].view(torch.int16))
    assert torch.equal(con["Vc"].view(torch.int16), ser["Vc"].view(torch.int16))
    assert torch.equal(out, ref_out)
    want = orc.decode_batch(inputs.as_f32(q, "bf16"), inputs.as_f32(Kc, "bf16"), inputs.as_f32(Vc, "bf16"),
                            lens, offs)
    assert np.max(np.abs(out.cpu().numpy() - want)) <= TOL_OUT["bf16"]


@pytest.mark.parametrize("graph", [False, True])
def test_gather_pipelined_beside_the_next_select(graph):
    """TB_EVICT_GATHER_CONCURRENT in the pipelined step: layer A's scores and
    selection, then layer B's scores and selection with, beside B's select,
    a decode over another cache and layer A's gather (both without
    dependency waits). Layer B is gathered last, as its own next step would.
    Indices and compacted caches bit-identical to tb_score_evict per layer,
    the decode output to its serial call; status words clean."""
    wl = inputs.WORKLOADS["7b"]
    lays = [inputs.make_layer(wl, li, alpha=0.5, n_override=[16384]) for li in (4, 5)]
    descs = [evict_desc(wl, lay, flags=tb.TB_EVICT_GATHER_CONCURRENT) for lay in lays]
    plain = [evict_desc(wl, lay) for lay in lays]
    # serial reference: one tb_score_evict per layer (the flag is ignored there)
    refs = []
    for lay, dsc, pl in zip(lays, descs, plain):
        r = _eviction_buffers(wl, lay, pl)
        tb.tb_score_evict(pl, r["q_win"], r["K"], r["V"], r["idx"], r["Kc"], r["Vc"], None, r["ws"])
        f = _eviction_buffers(wl, lay, dsc)
        tb.tb_score_evict(dsc, f["q_win"], f["K"], f["V"], f["idx"], f["Kc"], f["Vc"], None, f["ws"])
        torch.cuda.synchronize()
        assert tb.tb_read_status(r["ws"]) == (tb.TB_OK, 0)
        assert torch.equal(f["idx"], r["idx"])
        assert torch.equal(f["Kc"].view(torch.int16), r["Kc"].view(torch.int16))
        refs.append(r)
    caps = [int(plain[0].out_cap[0]) + 64]
    offs, rows, q, Kc, Vc = _cache(9, "bf16", wl.hq, wl.hkv, wl.head_dim, caps)
    lens_d = torch.tensor([caps[0] - 3], dtype=torch.int32, device="cuda")
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    ddesc = tb.DecodeDesc(hq=wl.hq, hkv=wl.hkv, head_dim=wl.head_dim, dtype=tb.TB_BF16,
                          cache_offset=offs, cache_cap=caps, cache_rows=rows, max_len=caps[0],
                          flags=tb.TB_DECODE_EARLY_CACHE_READ | tb.TB_DECODE_CONCURRENT,
                          max_ctas=sms - tb.tb_select_ctas(descs[1]))
    qd, Kd, Vd = to_dev(q, "bf16"), to_dev(Kc, "bf16"), to_dev(Vc, "bf16")
    dws = torch.empty(tb.tb_decode_workspace_size(ddesc), dtype=torch.uint8, device="cuda")
    tb.tb_decode_workspace_prepare(ddesc, dws)
    ref_out = torch.empty((1, wl.hq, wl.head_dim), dtype=torch.float32, device="cuda")
    tb.tb_decode_attn_prepared(ddesc, qd, Kd, Vd, lens_d, ref_out, dws)

    bufs = [_eviction_buffers(wl, lay, dsc) for lay, dsc in zip(lays, descs)]
    A, B = bufs
    out = torch.full_like(ref_out, float("nan"))
    main = torch.cuda.Stream()
    torch.cuda.synchronize()
    with torch.cuda.stream(main):
        tb.tb_window_scores(descs[0], A["q_win"], A["K"], A["scores"], A["ws"], stream=main)
        tb.tb_select_topk(descs[0], A["scores"], A["idx"], None, A["ws"], stream=main)
    main.synchronize()

    def step():
        tb.tb_window_scores(descs[1], B["q_win"], B["K"], B["scores"], B["ws"], stream=main)
        tb.tb_select_topk(descs[1], B["scores"], B["idx"], None, B["ws"], stream=main)
        tb.tb_decode_attn_prepared(ddesc, qd, Kd, Vd, lens_d, out, dws, stream=main)
        tb.tb_gather_kv(descs[0], A["idx"], A["K"], A["V"], A["Kc"], A["Vc"], stream=main)

    if graph:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=main):
            step()
        with torch.cuda.stream(main):
            g.replay()
    else:
        step()
    main.synchronize()
    tb.tb_gather_kv(plain[1], B["idx"], B["K"], B["V"], B["Kc"], B["Vc"])
    torch.cuda.synchronize()
    for buf, r in zip(bufs, refs):
        assert tb.tb_read_status(buf["ws"]) == (tb.TB_OK, 0)
        assert torch.equal(buf["idx"], r["idx"])
        assert torch.equal(buf["Kc"].view(torch.int16), r["Kc"].view(torch.int16))
        assert torch.equal(buf["Vc"].view(torch.int16), r["Vc"].view(torch.int16))
    assert tb.tb_read_status(dws) == (tb.TB_OK, 0)
    assert torch.equal(out, ref_out)
