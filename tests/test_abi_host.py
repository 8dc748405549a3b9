"""Host-side checks of the C ABI: the library loads, exports every symbol the
header declares, and rejects bad arguments before touching a GPU.

No test here launches device work: every call either queries sizes or fails
validation, which the library performs before its first CUDA call.
"""
import ctypes
import os
import re

import numpy as np
import pytest

from oracle import timebill_oracle as orc

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "timebill_kv.h")


@pytest.fixture(scope="session")
def tb():
    from paper_2512_21859_gb300 import build, binding
    build.build()
    binding.load()
    return binding


def _declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(tb_[a-z0-9_]+)\s*\(", text)))


def test_exports_every_declared_symbol(tb):
    names = _declared_functions()
    assert len(names) >= 14, names
    lib = ctypes.CDLL(tb.library_path())
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing


def _header_constants():
    """NAME -> value of the header's integer #defines and enum members."""
    text = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    consts = {}
    for name, val in re.findall(r"^#define\s+(TB_[A-Z0-9_]+)\s+(.+?)\s*$", text, flags=re.M):
        m = re.fullmatch(r"\(?\s*(\d+)u?\s*(?:<<\s*(\d+))?\s*\)?", val)
        assert m, (name, val)
        consts[name] = int(m.group(1)) << int(m.group(2) or 0)
    for name, val in re.findall(r"\b(TB_[A-Z0-9_]+)\s*=\s*(\d+)", text):
        consts[name] = int(val)
    return consts


def test_binding_constants_match_the_header(tb):
    consts = _header_constants()
    assert {"TB_OK", "TB_ERR_TIMEOUT", "TB_BF16", "TB_MAX_BATCH", "TB_EVICT_GATHER_CONCURRENT",
            "TB_DECODE_CONCURRENT", "TB_NOALLOC_SCRATCH_BYTES"} <= set(consts)
    for name, val in consts.items():
        assert getattr(tb, name) == val, name


def test_binding_structs_match_the_header(tb, tmp_path):
    """Every field of the header's structs sits at the offset the ctypes
    layout gives it, and the sizes agree (a C compiler reads the header)."""
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    pairs = [("tb_evict_desc", tb._EvictDescC), ("tb_decode_desc", tb._DecodeDescC),
             ("tb_time_model", tb.TimeModel)]
    lines = ["#include <stddef.h>", "#include <stdio.h>", '#include "timebill_kv.h"', "int main(void) {"]
    for cname, py in pairs:
        lines.append('  printf("%s sizeof %%zu\\n", sizeof(%s));' % (cname, cname))
        for field, _ in py._fields_:
            lines.append('  printf("%s %s %%zu\\n", offsetof(%s, %s));' % (cname, field, cname, field))
    lines += ["  return 0;", "}"]
    src, exe = tmp_path / "layout.c", tmp_path / "layout"
    src.write_text("\n".join(lines) + "\n")
    subprocess.run([cc, "-std=c11", "-I", os.path.dirname(HEADER), str(src), "-o", str(exe)], check=True)
    got = {}
    for line in subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.splitlines():
        cname, field, val = line.split()
        got[(cname, field)] = int(val)
    for cname, py in pairs:
        assert got[(cname, "sizeof")] == ctypes.sizeof(py), cname
        for field, _ in py._fields_:
            assert got[(cname, field)] == getattr(py, field).offset, (cname, field)


def _prototypes():
    """name -> (return type, [parameter declarations]) of the header's functions."""
    text = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    out = {}
    for ret, name, args in re.findall(r"([A-Za-z_][\w \*]*?)\s*\b(tb_[a-z0-9_]+)\s*\(([^;{]*?)\)\s*;",
                                      text, flags=re.S):
        params = [a.strip() for a in args.replace("\n", " ").split(",")] if args.strip() not in ("", "void") else []
        out[name] = (" ".join(ret.split()), params)
    return out


def _is_pointer_type(t):
    return t in (ctypes.c_void_p, ctypes.c_char_p) or issubclass(t, ctypes._Pointer) or hasattr(t, "_dtype_")


_SCALARS = {"int32_t": ctypes.c_int32, "int64_t": ctypes.c_int64, "uint64_t": ctypes.c_uint64,
            "size_t": ctypes.c_size_t, "double": ctypes.c_double, "tb_status": ctypes.c_int32}


def test_binding_signatures_match_the_header(tb):
    """Each entry point's ctypes argument list has the header's arity, a
    pointer where the header has a pointer or a stream, and the header's
    scalar type elsewhere; likewise the return type."""
    protos = _prototypes()
    assert set(protos) == set(_declared_functions())
    lib = tb.load()
    for name, (ret, params) in protos.items():
        fn = getattr(lib, name)
        assert fn.argtypes is not None and len(fn.argtypes) == len(params), name
        for decl, t in zip(params, fn.argtypes):
            if "*" in decl or decl.startswith("tb_stream_t"):
                assert _is_pointer_type(t), (name, decl, t)
            else:
                ctype = decl.replace("const ", "").split()[0]
                assert t is _SCALARS[ctype], (name, decl, t)
        if "*" in ret:
            assert fn.restype is ctypes.c_char_p, name
        else:
            assert fn.restype is _SCALARS[ret.split()[-1]], (name, ret)


def test_status_strings_and_version(tb):
    for s in range(6):
        assert tb.tb_status_string(s)
    assert tb.tb_status_string(99) == "unknown status"
    assert tb.tb_abi_version() == 103
    assert tb.tb_last_error_detail() == ""


def test_retained_count_matches_oracle(tb):
    for n in (1, 2, 17, 512, 4096, 32768, 131072, 10):
        for w in (1, 16, 64):
            if w > n:
                continue
            for a in np.concatenate([np.linspace(0, 1, 41), [0.3, 0.9, 0.95, 2 / 3]]):
                assert tb.tb_retained_count(n, w, float(a)) == orc.retained_count(n, w, float(a))


@pytest.mark.parametrize("n,w,a", [(10, 0, 0.5), (5, 6, 0.5), (10, 2, -0.1), (10, 2, 1.5),
                                   (10, 2, float("nan")), (10, 2, float("inf"))])
def test_retained_count_rejects(tb, n, w, a):
    with pytest.raises(tb.TbError) as e:
        tb.tb_retained_count(n, w, a)
    assert e.value.status == tb.TB_ERR_INVALID_ARG


def _desc(tb, **kw):
    base = dict(hq=4, hkv=2, head_dim=64, window=16, pool_k=7, dtype=tb.TB_F32, n=[512], alpha=[0.5])
    base.update(kw)
    return tb.EvictDesc(**base)


def test_layout_and_workspace(tb):
    d = _desc(tb, n=[512, 100, 40], alpha=[0.5, 0.0, 1.0])
    s, i = tb.tb_evict_layout(d)
    assert s == (512 - 16) + (100 - 16) + (40 - 16)
    assert i == sum(orc.retained_count(n, 16, a)[1] for n, a in [(512, .5), (100, 0), (40, 1)])
    ws = tb.tb_evict_workspace_size(d)
    assert ws > 256 and ws % 256 == 0
    d2 = _desc(tb, n=[4096])
    assert tb.tb_evict_workspace_size(d2) > tb.tb_evict_workspace_size(_desc(tb, n=[512]))


@pytest.mark.parametrize("kw,status", [
    (dict(hq=5), 1),                         # hq not a multiple of hkv
    (dict(head_dim=96), 2),
    (dict(dtype=7), 2),
    (dict(pool_k=4), 1),
    (dict(pool_k=65), 1),
    (dict(window=0), 1),
    (dict(n=[8]), 1),                        # n < window
    (dict(alpha=[1.5]), 1),
    (dict(alpha=[float("nan")]), 1),
    (dict(kv_rows=100), 1),                  # request rows beyond kv_rows
    (dict(kv_offset=[-1]), 1),
    (dict(out_cap=[100]), 1),                # out_cap < R
    (dict(out_rows=10), 1),
    (dict(flags=8), 1),                      # a flag bit the library does not know
    (dict(n=[512] * 65, alpha=[0.5] * 65), 2),  # batch > TB_MAX_BATCH
    (dict(hq=2048, hkv=1), 2),               # G*W beyond the supported window rows
])
def test_evict_desc_rejects(tb, kw, status):
    d = _desc(tb, **kw)
    with pytest.raises(tb.TbError) as e:
        tb.tb_evict_layout(d)
    assert e.value.status == status


def test_overlapping_outputs_rejected(tb):
    d = _desc(tb, n=[512, 512], alpha=[0.5, 0.5], out_offset=[0, 100], out_cap=[272, 272], out_rows=1000)
    with pytest.raises(tb.TbError) as e:
        tb.tb_evict_layout(d)
    assert e.value.status == tb.TB_ERR_INVALID_ARG


def test_calls_fail_before_any_launch(tb):
    d = _desc(tb)
    ws_bytes = tb.tb_evict_workspace_size(d)
    fake = 1 << 20   # a 256-aligned address that is never dereferenced
    # null tensors
    for args in [(0, fake, fake), (fake, 0, fake), (fake, fake, 0)]:
        with pytest.raises(tb.TbError) as e:
            tb.tb_window_scores(d, *args, fake, ws_bytes, stream=0)
        assert e.value.status == tb.TB_ERR_INVALID_ARG
    # misaligned tensor
    with pytest.raises(tb.TbError) as e:
        tb.tb_score_evict(d, fake + 8, fake, fake, fake, fake, fake, None, fake, ws_bytes, stream=0)
    assert e.value.status == tb.TB_ERR_INVALID_ARG
    # workspace: missing, too small, misaligned
    for w, wb in [(0, ws_bytes), (fake, ws_bytes - 1), (fake + 16, ws_bytes)]:
        with pytest.raises(tb.TbError) as e:
            tb.tb_score_evict(d, fake, fake, fake, fake, fake, fake, None, w, wb, stream=0)
        assert e.value.status == tb.TB_ERR_WORKSPACE
        with pytest.raises(tb.TbError) as e:
            tb.tb_select_topk(d, fake, fake, None, w, wb, stream=0)
        assert e.value.status == tb.TB_ERR_WORKSPACE
    with pytest.raises(tb.TbError) as e:
        tb.tb_gather_kv(d, fake, fake, 0, fake, fake, stream=0)
    assert e.value.status == tb.TB_ERR_INVALID_ARG


def _ddesc(tb, **kw):
    base = dict(hq=28, hkv=4, head_dim=128, dtype=tb.TB_BF16, cache_offset=[0], cache_cap=[5000],
                cache_rows=5000, max_len=4096)
    base.update(kw)
    return tb.DecodeDesc(**base)


def test_decode_workspace(tb):
    a = tb.tb_decode_workspace_size(_ddesc(tb))
    b = tb.tb_decode_workspace_size(_ddesc(tb, cache_offset=[0, 5000], cache_cap=[5000, 5000], cache_rows=10000))
    assert a > 256 and b >= a


def test_decode_cta_budget_shrinks_the_splits(tb):
    """A CTA budget gives fewer splits, so the split partials (and the
    workspace) shrink; flags with the concurrency bit are accepted."""
    full = tb.tb_decode_workspace_size(_ddesc(tb))
    assert tb.tb_decode_workspace_size(_ddesc(tb, max_ctas=152)) == full
    prev = full
    for m in (88, 40, 8, 4, 1):
        w = tb.tb_decode_workspace_size(_ddesc(tb, max_ctas=m, flags=tb.TB_DECODE_CONCURRENT))
        assert w <= prev
        prev = w
    assert prev < full
    # a budget below one CTA per (request, KV head) still gives one split each
    assert tb.tb_decode_workspace_size(_ddesc(tb, max_ctas=1)) == tb.tb_decode_workspace_size(
        _ddesc(tb, max_ctas=4))


@pytest.mark.parametrize("n,w,hkv,batch,want", [
    (512, 16, 2, 1, 2),              # prefix 496: one CTA per cluster
    (4096 + 16, 16, 2, 1, 2),        # 4096 prefix keys: still one
    (4096 + 17, 16, 2, 1, 4),        # one more key: two per cluster
    (32768, 32, 4, 1, 32),           # 32K prefix: eight per cluster
    (131072, 64, 8, 1, 64),          # 128K: eight per cluster, eight KV heads
    (131072, 64, 8, 2, 128),         # two requests
])
def test_select_ctas(tb, n, w, hkv, batch, want):
    d = tb.EvictDesc(hq=4 * hkv, hkv=hkv, head_dim=64, window=w, pool_k=7, dtype=tb.TB_F32,
                     n=[n] * batch, alpha=[0.5] * batch)
    assert tb.tb_select_ctas(d) == want


def test_select_ctas_fallback_and_errors(tb):
    # a prefix longer than eight 16K slices runs the one-CTA-per-segment fallback
    d = tb.EvictDesc(hq=4, hkv=2, head_dim=64, window=16, pool_k=7, dtype=tb.TB_F32,
                     n=[8 * 16384 + 100], alpha=[0.5])
    assert tb.tb_select_ctas(d) == 2
    with pytest.raises(tb.TbError) as e:
        tb.tb_select_ctas(_desc(tb, hq=5))
    assert e.value.status == tb.TB_ERR_INVALID_ARG


@pytest.mark.parametrize("kw,status", [
    (dict(hq=30), 1),
    (dict(head_dim=80), 2),
    (dict(dtype=3), 2),
    (dict(out_dtype=1, dtype=0), 2),   # bf16 output of fp32 inputs
    (dict(max_len=0), 1),
    (dict(cache_rows=100), 1),
    (dict(cache_offset=[-4]), 1),
    (dict(hq=132, hkv=4), 2),                   # group of 33 heads at d=128
    (dict(flags=4), 1),                         # an undefined flag bit
    (dict(max_ctas=-1), 1),                     # a negative CTA budget
])
def test_decode_desc_rejects(tb, kw, status):
    with pytest.raises(tb.TbError) as e:
        tb.tb_decode_workspace_size(_ddesc(tb, **kw))
    assert e.value.status == status


def test_decode_call_fails_before_launch(tb):
    d = _ddesc(tb)
    wb = tb.tb_decode_workspace_size(d)
    fake = 1 << 20
    with pytest.raises(tb.TbError) as e:
        tb.tb_decode_attn(d, fake, fake, fake, 0, fake, fake, wb, stream=0)
    assert e.value.status == tb.TB_ERR_INVALID_ARG
    with pytest.raises(tb.TbError) as e:
        tb.tb_decode_attn(d, fake, fake, fake, fake, fake, fake, wb - 1, stream=0)
    assert e.value.status == tb.TB_ERR_WORKSPACE


def test_prepared_decode_calls_fail_before_launch(tb):
    d = _ddesc(tb)
    wb = tb.tb_decode_workspace_size(d)
    fake = 1 << 20
    with pytest.raises(tb.TbError) as e:
        tb.tb_decode_attn_prepared(d, fake, fake, fake, 0, fake, fake, wb, stream=0)
    assert e.value.status == tb.TB_ERR_INVALID_ARG
    with pytest.raises(tb.TbError) as e:
        tb.tb_decode_attn_prepared(d, fake, fake, fake, fake, fake, fake, wb - 1, stream=0)
    assert e.value.status == tb.TB_ERR_WORKSPACE
    with pytest.raises(tb.TbError) as e:
        tb.tb_decode_workspace_prepare(d, fake, wb - 1, stream=0)
    assert e.value.status == tb.TB_ERR_WORKSPACE
    with pytest.raises(tb.TbError) as e:
        tb.tb_decode_workspace_prepare(_ddesc(tb, hq=30), fake, wb, stream=0)
    assert e.value.status == tb.TB_ERR_INVALID_ARG
