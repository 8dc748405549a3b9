#!/usr/bin/env python
"""Benchmark of TimeBill's eviction + decode-attention hot path on GB300.

One step = one transformer layer of the path: one decode step of attention
over a compacted cache (tb_decode_attn_prepared: the decode workspace is
prepared once, as a decode loop keeps it) and a layer's prompt-time
eviction (tb_window_scores -> tb_select_topk -> tb_gather_kv, the stages
tb_score_evict chains), pipelined over the layer rotation: step i scores
layer i and selects its rows, and beside that select run the decode over
layer i-2's compacted cache and the gather of layer i-1, both without
dependency waits (TB_DECODE_CONCURRENT with a CTA budget,
TB_EVICT_GATHER_CONCURRENT). --serial-step: decode first, then the eviction,
on one stream. Layers rotate over enough device buffers that every step's
inputs are larger than L2 (129 MB), so no step reads another step's data
from cache.

Prints ONE JSON line. value = algorithmic HBM bytes of the step (K read once
to score, retained K/V rows read and written, compacted K/V read by decode)
per second, in GB/s, summed over ranks. Under torchrun every rank runs its
own replica (independent layers: the path has no cross-rank exchange).

``--impl reference`` times the CPU fp64 oracle instead (the method's only
reference; no GPU work) on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2512_21859_gb300 import inputs  # noqa: E402

METRIC = "evict + decode-attn µs/layer and HBM GB/s (fraction of ~8 TB/s) vs α"
L2_BYTES = 129e6
NOMINAL_HBM_GBS = 8000.0
# the metric's alpha axis, carried in the one JSON line of every run
ALPHA_SWEEP = [("128k", (0.5, 0.75, 0.9)), ("32k", (0.0, 0.25, 0.5, 0.75, 0.9, 0.95))]
# the algorithmic bytes of each stage per launch (the method's minimum)
ALG_BYTES_RULE = {
    "window_scores": "e Hkv d sum(N) + q_win bytes: K read once",
    "select_topk": "4 Hkv (2 sum(P) + sum(R)): scores read, pooled written, indices written",
    "gather_kv": "4 e Hkv d sum(R): retained K and V rows read and written",
    "decode_attn": "2 e Hkv d sum(len) + B Hq d (e + 4): compacted K and V read, query read, fp32 output",
}


def parse_args(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="128k", choices=sorted(inputs.WORKLOADS))
    ap.add_argument("--alpha", type=float, default=None,
                    help="eviction ratio for every request (default: the workload's own)")
    ap.add_argument("--sweep", default=None,
                    help="comma-separated alphas: print one line per alpha")
    ap.add_argument("--e2e-steps", type=int, default=None)
    ap.add_argument("--no-variants", action="store_true",
                    help="skip timing tb_window_scores_lse beside the step (its line is then null)")
    ap.add_argument("--fit-time-model", action="store_true",
                    help="profile tb_decode_attn_prepared over N_kv and tb_score_evict over N_x on the 7b "
                         "shape and print the least-squares time model (Eq. 6a/6b) with its MAPE")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--serial-step", action="store_true",
                    help="run the step's decode before the eviction (default: between the select and "
                         "the gather, so that its CTAs start during the select)")
    ap.add_argument("--no-alpha-sweep", action="store_true",
                    help="skip the per-alpha stage table (128K at 0.5/0.75/0.9, 32K at 0..0.95)")
    ap.add_argument("--sweep-steps", type=int, default=12,
                    help="launches per stage timing of each alpha point")
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="target seconds of oracle work for the cpu_baseline sample")
    return ap.parse_args(argv)


# ---------------------------------------------------------------------------
# algorithmic bytes (the method's minimum traffic per layer)
# ---------------------------------------------------------------------------

def elem_bytes(wl):
    return 4 if wl.dtype == "f32" else 2


def retained(n, window, alpha):
    from paper_2512_21859_gb300 import binding as tb
    return tb.tb_retained_count(int(n), int(window), float(alpha))


def alg_bytes(wl, n, alpha, lens):
    """Per-layer algorithmic bytes of each stage (HBM, minimum)."""
    e = elem_bytes(wl)
    row = e * wl.head_dim
    B = len(n)
    R = [retained(nb, wl.window, a)[1] for nb, a in zip(n, alpha)]
    P = [int(nb) - wl.window for nb in n]
    q_win = B * wl.hq * wl.window * wl.head_dim * e
    scores = row * wl.hkv * int(np.sum(n)) + q_win
    select = 4 * wl.hkv * (2 * int(np.sum(P)) + int(np.sum(R)))
    gather = 4 * row * wl.hkv * int(np.sum(R))
    decode = 2 * row * wl.hkv * int(np.sum(lens)) + B * wl.hq * wl.head_dim * (e + 4)
    evict_min = row * wl.hkv * int(np.sum(n) + 4 * np.sum(R)) + q_win
    return {"window_scores": scores, "select_topk": select, "gather_kv": gather,
            "decode_attn": decode, "evict": evict_min, "step": evict_min + decode, "R": R}


def stage_rooflines(wl, n, ab, stage_ms, peaks):
    """Every stage against its HBM roofline: algorithmic bytes over the
    stage's per-launch time against the measured copy bandwidth. The window
    scoring is also a dense bf16 contraction; beside its HBM fraction it
    reports the tensor rate on the method's flops (one Q K^T over the N keys
    of every window row, 2 Hq W d N) and on the flops this kernel executes
    (two passes: N keys for the row statistics, then the P = N - W prefix
    keys for the sums), both against the measured burst bf16 rate (the
    stage is timed alone, in graphs of a few hundred microseconds)."""
    hbm = float(peaks["hbm_gbs"])
    out = {}
    for s, ms in stage_ms.items():
        gbs = ab[s] / (ms * 1e-3) / 1e9
        out[s] = {"bound": "hbm", "alg_bytes": int(ab[s]), "us": round(1e3 * ms, 2),
                  "achieved_gbs": round(gbs, 1), "frac": round(gbs / hbm, 4)}
    if "window_scores" in stage_ms and wl.dtype == "bf16":
        per_key = 2.0 * wl.hq * wl.window * wl.head_dim
        method = per_key * float(np.sum(n))
        executed = per_key * float(2 * np.sum(n) - len(n) * wl.window)
        sec = stage_ms["window_scores"] * 1e-3
        peak = float(peaks["bf16_tflops"])
        out["window_scores"]["tensor"] = {
            "flops": method, "achieved_tflops": round(method / sec / 1e12, 1), "peak_tflops": peak,
            "frac": round(method / sec / 1e12 / peak, 4),
            "flops_rule": "the method's contraction: 2 Hq W d flops per key, one pass over the N keys",
            "executed_flops": executed, "executed_tflops": round(executed / sec / 1e12, 1),
            "executed_frac": round(executed / sec / 1e12 / peak, 4),
            "executed_rule": "two passes as the kernel runs them: N keys (row statistics) + N - W keys (sums)",
            "peak_source": "measured burst bf16 (MEASURED_PEAKS.json bf16_tflops): the stage is timed alone"}
    return out


# ---------------------------------------------------------------------------
# distributed plumbing
# ---------------------------------------------------------------------------

def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def dist_init(world, use_cuda):
    if world <= 1:
        return None
    import torch.distributed as dist
    dist.init_process_group(backend="nccl" if use_cuda else "gloo")
    return dist


def max_over_ranks(dist, value, device=None):
    """The largest of every rank's `value`: the job's time is its slowest rank's."""
    if not dist:
        return float(value)
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_value(world, step_bytes, steps, total_ms):
    """Whole-job GB/s: every rank moved step_bytes per step (weak scaling)."""
    return world * step_bytes * steps / (total_ms * 1e-3) / 1e9


# ---------------------------------------------------------------------------
# clocks sampled during the timed region
# ---------------------------------------------------------------------------

REASONS = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]


class ClockSampler:
    def __init__(self, gpu_index: int):
        self.proc = None
        # the samples go to a file of their own; the BENCH_CLOCKS_DIR
        # environment variable keeps them, else a temporary directory
        out_dir = os.environ.get("BENCH_CLOCKS_DIR") or tempfile.gettempdir()
        self.path = os.path.join(out_dir, "clocks_bench_%d.csv" % os.getpid())
        q = "index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active," + ",".join(
            "clocks_event_reasons." + r for r in REASONS)
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(gpu_index), "--query-gpu=" + q,
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=self.f, stderr=subprocess.DEVNULL)
        except (OSError, ValueError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.close()
        sm, mx, active = [], [], set()
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 5 + len(REASONS):
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx.append(float(parts[2]))
                except ValueError:
                    continue
                for r, v in zip(REASONS, parts[5:]):
                    if v.lower().startswith("active"):
                        active.add(r)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(active)}


# ---------------------------------------------------------------------------
# profile-derived DRAM traffic (ncu), used only while the kernel source matches
# ---------------------------------------------------------------------------

def kernel_source_digest(files):
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, "paper_2512_21859_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def profiled_traffic(stage, workload):
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        table = json.load(f)
    ent = table.get("%s/%s" % (stage, workload))
    if not ent:
        return None
    try:
        if kernel_source_digest(ent["sources"]) != ent["source_digest"]:
            return None
    except OSError:
        return None
    return ent["dram_bytes_per_launch"]


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------

STAGES = ["decode_attn", "window_scores", "select_topk", "gather_kv"]


def pipelined_step(i, L):
    """The C-ABI calls of step i of the pipelined layer loop over L >= 2
    layer buffers, in stream order, as (call, buffer): layer i's scores and
    select, then beside that select the decode over the cache compacted two
    steps earlier and the gather of the rows selected one step earlier."""
    return [("window_scores", i % L), ("select_topk", i % L),
            ("decode_beside_select", (i + L - 2) % L), ("gather_beside_select", (i + L - 1) % L)]


def to_device(torch, wl, x, dev):
    if wl.dtype == "bf16":
        return torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).view(torch.bfloat16).to(dev)
    return torch.from_numpy(np.ascontiguousarray(x)).to(dev)


def load_workload(torch, wl, rank, dev):
    """One layer's eviction inputs on the device, cloned into enough
    rotating buffers that their K and V together exceed L2 three times
    over. The inputs do not depend on alpha (it only sets the budget)."""
    lay = inputs.make_layer(wl, rank)
    n = lay["n"]
    layer_bytes = 2 * wl.hkv * int(np.sum(n)) * wl.head_dim * elem_bytes(wl)
    L = int(min(64, max(2, math.ceil(3 * L2_BYTES / layer_bytes))))
    base = {k: to_device(torch, wl, lay[k], dev) for k in ("q_win", "K", "V")}
    layers = [{k: (v if li == 0 else v.clone()) for k, v in base.items()} for li in range(L)]
    return {"wl": wl, "lay": lay, "n": n, "L": L, "layer_bytes": layer_bytes, "layers": layers}


def setup_alpha(torch, tb, W, alpha_vec, rank, dev, stream):
    """Descriptors and per-buffer outputs of one eviction ratio; runs every
    stage once per buffer (filling each compacted cache) and checks the
    status words. The decode stage gets its own rotation of compacted caches
    (copies of the buffers' own) large enough that one replay of its graph
    reads more than three times L2."""
    wl, n, lay = W["wl"], W["n"], W["lay"]
    B = len(n)
    R = [retained(nb, wl.window, x)[1] for nb, x in zip(n, alpha_vec)]
    lens_h = [r + 1 for r in R]
    ab = alg_bytes(wl, n, alpha_vec, lens_h)
    desc = tb.EvictDesc(hq=wl.hq, hkv=wl.hkv, head_dim=wl.head_dim, window=wl.window,
                        pool_k=wl.pool_k, dtype=tb.TB_BF16 if wl.dtype == "bf16" else tb.TB_F32,
                        n=n, alpha=alpha_vec, kv_offset=lay["kv_offset"], kv_rows=int(np.sum(n)),
                        out_cap=lens_h)
    # the step's gather runs beside the next layer's select (no dependency wait before its copies)
    gdesc = tb.EvictDesc(hq=wl.hq, hkv=wl.hkv, head_dim=wl.head_dim, window=wl.window,
                         pool_k=wl.pool_k, dtype=desc.dtype, n=n, alpha=alpha_vec, kv_offset=lay["kv_offset"],
                         kv_rows=int(np.sum(n)), out_cap=lens_h, flags=tb.TB_EVICT_GATHER_CONCURRENT)
    score_rows, idx_rows = tb.tb_evict_layout(desc)
    # the step's own K/V row is in place before the decode, and the kernel
    # before each decode writes no row of its cache: the early-read assertion holds
    ddesc = tb.DecodeDesc(hq=wl.hq, hkv=wl.hkv, head_dim=wl.head_dim, dtype=desc.dtype,
                          cache_offset=desc.out_offset, cache_cap=desc.out_cap,
                          cache_rows=desc.out_rows, max_len=max(lens_h), flags=tb.TB_DECODE_EARLY_CACHE_READ)
    # the step's decode runs beside the select (TB_DECODE_CONCURRENT) on
    # part of the SMs the select leaves free, the rest left to the gather
    # beside it: 0.6 of them (measured on GB300, CTA budgets at 128K 88 /
    # 72 / 56 / 40: step 140.6 / 139.8 / 140.0 / 141.3 us; at 32K 120 / 96 /
    # 72 / 48: 47.3 / 46.7 / 45.8 / 48.6 us; as fractions of the free SMs,
    # 0.4 / 0.5 / 0.6 / 0.7 / 0.8 at 128K: 144.2 / 139.6 / 136.6 / 136.6 /
    # 136.5 us, at 32K: 44.7 / 42.8 / 42.4 / 42.4 / 42.4 us); its own
    # descriptor and prepared workspaces
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    free = sms - tb.tb_select_ctas(desc)
    # a select that fills the GPU (many requests): the default split
    step_ctas = int(0.6 * free + 0.5) if free >= sms // 4 else 0
    sddesc = tb.DecodeDesc(hq=wl.hq, hkv=wl.hkv, head_dim=wl.head_dim, dtype=desc.dtype,
                           cache_offset=desc.out_offset, cache_cap=desc.out_cap, cache_rows=desc.out_rows,
                           max_len=max(lens_h), flags=tb.TB_DECODE_EARLY_CACHE_READ | tb.TB_DECODE_CONCURRENT,
                           max_ctas=step_ctas)
    ews = tb.tb_evict_workspace_size(desc)
    dws = tb.tb_decode_workspace_size(ddesc)
    sdws = tb.tb_decode_workspace_size(sddesc)
    step_in = inputs.make_decode_step(wl, rank, 1, B)
    q_dec = to_device(torch, wl, step_in["q"], dev)
    kn, vn = to_device(torch, wl, step_in["k_new"], dev), to_device(torch, wl, step_in["v_new"], dev)
    bufs = []
    for lb in W["layers"]:
        d = dict(lb)
        d["Kc"] = torch.zeros((wl.hkv, desc.out_rows, wl.head_dim), dtype=lb["K"].dtype, device=dev)
        d["Vc"] = torch.zeros_like(d["Kc"])
        for b in range(B):   # the decode token's own K/V row, after the retained rows
            row = int(desc.out_offset[b]) + R[b]
            d["Kc"][:, row] = kn[:, b]
            d["Vc"][:, row] = vn[:, b]
        d["scores"] = torch.empty((wl.hkv, max(score_rows, 1)), dtype=torch.float32, device=dev)
        d["idx"] = torch.empty((wl.hkv, idx_rows), dtype=torch.int32, device=dev)
        d["ews"] = torch.empty(ews, dtype=torch.uint8, device=dev)
        d["dws"] = torch.empty(dws, dtype=torch.uint8, device=dev)
        tb.tb_decode_workspace_prepare(ddesc, d["dws"], stream=stream)
        d["sdws"] = torch.empty(sdws, dtype=torch.uint8, device=dev)
        tb.tb_decode_workspace_prepare(sddesc, d["sdws"], stream=stream)
        d["out"] = torch.empty((B, wl.hq, wl.head_dim), dtype=torch.float32, device=dev)
        bufs.append(d)
    lens = torch.tensor(lens_h, dtype=torch.int32, device=dev)

    def stage_call(name, d, st):
        if name == "decode_attn":
            tb.tb_decode_attn_prepared(ddesc, q_dec, d["Kc"], d["Vc"], lens, d["out"], d["dws"], stream=st)
        elif name == "decode_beside_select":
            tb.tb_decode_attn_prepared(sddesc, q_dec, d["Kc"], d["Vc"], lens, d["out"], d["sdws"], stream=st)
        elif name == "gather_beside_select":
            tb.tb_gather_kv(gdesc, d["idx"], d["K"], d["V"], d["Kc"], d["Vc"], stream=st)
        elif name == "window_scores":
            tb.tb_window_scores(desc, d["q_win"], d["K"], d["scores"], d["ews"], stream=st)
        elif name == "select_topk":
            tb.tb_select_topk(desc, d["scores"], d["idx"], None, d["ews"], stream=st)
        else:
            tb.tb_gather_kv(desc, d["idx"], d["K"], d["V"], d["Kc"], d["Vc"], stream=st)

    for d in bufs:
        for name in STAGES:
            stage_call(name, d, stream)
    torch.cuda.synchronize(dev)
    for d in bufs:
        st, raw = tb.tb_read_status(d["ews"], stream=stream)
        assert st == tb.TB_OK, raw
    # the decode's own rotation: each extra buffer a copy of a compacted cache
    # the eviction wrote, with its own prepared workspace
    Ld = int(min(64, max(len(bufs), math.ceil(3 * L2_BYTES / ab["decode_attn"]))))
    dec_bufs = list(bufs)
    for i in range(len(bufs), Ld):
        src = bufs[i % len(bufs)]
        d = {"Kc": src["Kc"].clone(), "Vc": src["Vc"].clone(),
             "dws": torch.empty(dws, dtype=torch.uint8, device=dev), "out": torch.empty_like(src["out"])}
        tb.tb_decode_workspace_prepare(ddesc, d["dws"], stream=stream)
        dec_bufs.append(d)
    torch.cuda.synchronize(dev)
    return {"desc": desc, "ddesc": ddesc, "bufs": bufs, "dec_bufs": dec_bufs, "R": R, "ab": ab,
            "stage_call": stage_call, "step_in": step_in, "ews": ews, "dws": dws, "step_ctas": step_ctas}


def check_decode_status(tb, stream, S):
    for d in S["dec_bufs"]:
        st, raw = tb.tb_read_status(d["dws"], stream=stream)
        assert st == tb.TB_OK, raw
    for d in S["bufs"]:
        st, raw = tb.tb_read_status(d["sdws"], stream=stream)
        assert st == tb.TB_OK, raw


def sweep_points(torch, tb, W, alphas, rank, dev, stream, peaks, steps):
    """The metric's alpha axis: per-stage device time per layer (each stage
    timed as in the headline) and the eviction and decode HBM fractions at
    each alpha, on the same rotated inputs."""
    wl = W["wl"]
    hbm = float(peaks["hbm_gbs"])
    cap = torch.cuda.Stream(dev)
    rows = []
    for alpha in alphas:
        avec = np.full(len(W["n"]), float(alpha))
        S = setup_alpha(torch, tb, W, avec, rank, dev, stream)
        ms, _ = time_stages(torch, dev, stream, cap, S, steps)
        check_decode_status(tb, stream, S)
        ab = S["ab"]
        ev_ms = ms["window_scores"] + ms["select_topk"] + ms["gather_kv"]
        ev_gbs = ab["evict"] / (ev_ms * 1e-3) / 1e9
        dec_gbs = ab["decode_attn"] / (ms["decode_attn"] * 1e-3) / 1e9
        rows.append({"workload": wl.name, "alpha": float(alpha), "R": int(S["R"][0]),
                     "us": {s: round(1e3 * v, 2) for s, v in ms.items()},
                     "evict_us": round(1e3 * ev_ms, 2), "evict_gbs": round(ev_gbs, 1),
                     "evict_frac": round(ev_gbs / hbm, 4), "decode_gbs": round(dec_gbs, 1),
                     "decode_frac": round(dec_gbs / hbm, 4),
                     "decode_rotation": len(S["dec_bufs"])})
        del S
        torch.cuda.empty_cache()
    return rows


def run_ours(args, wl, alpha, world, rank, local, dist):
    import torch
    from paper_2512_21859_gb300 import binding as tb

    torch.cuda.set_device(local)
    tb.load()
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream(dev)
    W = load_workload(torch, wl, rank, dev)
    n = W["n"]
    a = inputs.request_shapes(wl, alpha)[1]
    L = W["L"]
    S = setup_alpha(torch, tb, W, a, rank, dev, stream)
    ab, R, desc, ddesc = S["ab"], S["R"], S["desc"], S["ddesc"]
    stage_call = S["stage_call"]
    layers = S["bufs"]
    step_ctas = S["step_ctas"]

    # each layer buffer's step captured into a CUDA graph of the four calls,
    # pipelined over the layer rotation: step i scores layer i and selects
    # its rows; beside that select (bound by the latency of its phases on
    # the SMs its clusters hold) run, without waiting for it first, the decode
    # over layer i-2's compacted cache (TB_DECODE_CONCURRENT, a CTA budget
    # of the SMs the select leaves free) and the gather of layer i-1 (its
    # rows selected in step i-1; TB_EVICT_GATHER_CONCURRENT), both bound by
    # HBM. Nothing in the step writes what another call of it reads: the
    # gather writes layer i-1's compacted cache, the decode reads layer
    # i-2's (distinct buffers: at least two in the rotation). Every step
    # thus does one layer's scoring, select, gather and decode step.
    # --serial-step: the decode first, then the eviction, over the buffer's
    # own cache, on one stream.
    # A serving loop captures many layers in one graph; here one graph holds
    # a whole rotation (the L steps over the L buffers, in order), so that
    # K steps are K / L replays of it (a graph per step adds the gap between
    # graph launches to every step: 32K, a graph of the scoring alone,
    # 27.9 us per step against 24 us per launch inside one graph). Steps
    # left over when L does not divide K replay one-step graphs.
    assert L >= 2
    cap = torch.cuda.Stream(dev)

    def capture_step(i, d):
        if args.serial_step:
            for name in STAGES:
                stage_call(name, d, cap)
        else:
            for name, b in pipelined_step(i, L):
                stage_call(name, layers[b], cap)

    step_graphs = []
    kernels_per_step = None
    for i, d in enumerate(layers):
        g = torch.cuda.CUDAGraph()
        c0 = tb.tb_launch_counter()
        with torch.cuda.graph(g, stream=cap):
            capture_step(i, d)
        kernels_per_step = tb.tb_launch_counter() - c0
        step_graphs.append(g)
    rotation = torch.cuda.CUDAGraph()
    with torch.cuda.graph(rotation, stream=cap):
        for i, d in enumerate(layers):
            capture_step(i, d)
    torch.cuda.synchronize(dev)

    def run_steps(n):
        """n steps from the first buffer of the rotation on: whole-rotation
        graph replays, then one-step graphs for the rest."""
        for _ in range(n // L):
            rotation.replay()
        for i in range(n % L):
            step_graphs[i].replay()

    with torch.cuda.stream(stream):
        run_steps(max(args.warmup, L) // L * L + L)
    torch.cuda.synchronize(dev)

    K = args.steps
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(local)
    if dist:
        dist.barrier()
    torch.cuda.synchronize(dev)
    with torch.cuda.stream(stream):
        t0.record(stream)
        run_steps(K)
        t1.record(stream)
    torch.cuda.synchronize(dev)
    if dist:
        dist.barrier()
    total_ms = t0.elapsed_time(t1)
    stage_ms, stage_timing = time_stages(torch, dev, stream, cap, S, K)
    clocks = sampler.stop()
    launches = kernels_per_step * K
    total_ms = max_over_ranks(dist, total_ms, dev)
    check_decode_status(tb, stream, S)
    ms_step = total_ms / K
    value = job_value(world, ab["step"], K, total_ms)

    # roofline of the dominant stage: algorithmic HBM bytes per launch over
    # its per-launch time, against the measured copy bandwidth
    with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
        peaks = json.load(f)
    peak = float(peaks["hbm_gbs"])
    dom = max(STAGES, key=lambda s: stage_ms[s])
    achieved = ab[dom] / (stage_ms[dom] * 1e-3) / 1e9
    sroof = stage_rooflines(wl, n, ab, stage_ms, peaks)
    roof = {"kernel": dom, "bound": "hbm", "achieved": round(achieved, 1), "peak": peak,
            "unit": "GB/s", "frac": round(achieved / peak, 4),
            "peak_source": "measured (MEASURED_PEAKS.json hbm_gbs)",
            "traffic": profiled_traffic(dom, wl.name),
            "alg_bytes_per_launch": int(ab[dom]), "avg_launch_ms": round(stage_ms[dom], 5),
            "bytes_rule": ALG_BYTES_RULE.get(dom, "")}
    if "tensor" in sroof.get(dom, {}):
        roof["tensor"] = sroof[dom]["tensor"]

    lse_var = None if args.no_variants else time_lse_variant(torch, tb, dev, stream, wl, W["lay"], desc, layers,
                                                             stage_ms, ms_step, n, peaks, ab["evict"])

    e2e = run_e2e(args, wl, tb, torch, dev, stream, W["lay"], desc, ddesc, S["ews"], S["dws"], S["step_in"],
                  ab, R)

    sweep = None
    if not args.no_alpha_sweep:
        del S, layers, step_graphs, stage_call
        torch.cuda.empty_cache()
        sweep = {"timing": "per stage as in stage_timing; each alpha on the same rotated inputs",
                 "points": []}
        for wname, alphas in ALPHA_SWEEP:
            Wx = W if wname == wl.name else load_workload(torch, inputs.WORKLOADS[wname], rank, dev)
            sweep["points"] += sweep_points(torch, tb, Wx, alphas, rank, dev, stream, peaks,
                                            args.sweep_steps)
            if Wx is not W:
                del Wx
                torch.cuda.empty_cache()

    evict_us = 1e3 * (stage_ms["window_scores"] + stage_ms["select_topk"] + stage_ms["gather_kv"])
    res = {
        "metric": METRIC, "value": round(value, 1), "unit": "GB/s", "n_gpus": world,
        "steps": K, "warmup": args.warmup, "ms_per_step": round(ms_step, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": wl.dtype, "data": "synthetic (seeded Gaussian q/K/V with planted heavy hitters)",
        "config": {
            "workload": describe(wl, n, a), "alpha": float(a[0]) if len(set(a.tolist())) == 1 else a.tolist(),
            "layers_rotated": L, "l2": "inputs larger than L2: %d rotating layer buffers of %.0f MB" % (
                L, W["layer_bytes"] / 1e6),
            "step": "one layer's window_scores + select_topk + gather_kv + decode_attn (one token); "
                    "pipelined, the gather and the decode are of the previous layers (see launch)",
            "decode_call": "tb_decode_attn_prepared with TB_DECODE_EARLY_CACHE_READ (workspace prepared once; "
                           "no per-call clearing kernel; first tiles requested before the preceding kernel ends); "
                           "in the step also with TB_DECODE_CONCURRENT and max_ctas (no dependency wait before its "
                           "work: it runs beside the select)",
            "launch": "the steps replay a CUDA graph of a whole rotation of %d steps (one-step graphs for "
                      "any remainder of the K steps), each step the four C-ABI calls" % L + (
                ": decode_attn, window_scores, select_topk, gather_kv" if args.serial_step else
                ", pipelined over the layer rotation: step i runs window_scores and select_topk of "
                "layer i, and beside that select, without waiting for it first, the decode over layer i-2's "
                "compacted cache (TB_DECODE_CONCURRENT, max_ctas = %s) and the gather of layer i-1 "
                "(TB_EVICT_GATHER_CONCURRENT)" % ("0.6 x (SMs - tb_select_ctas) = %d" % step_ctas if step_ctas
                                                   else "0: the select fills the GPU")),
            "stage_timing": stage_timing,
            "parallelism": "replicas" if world > 1 else "single GPU"},
        "us_per_layer": {"evict": round(evict_us, 2), "decode": round(1e3 * stage_ms["decode_attn"], 2),
                         "step": round(1e3 * ms_step, 2),
                         "stages": {s: round(1e3 * v, 2) for s, v in stage_ms.items()}},
        "gbs": {"evict": round(ab["evict"] / (evict_us * 1e-6) / 1e9, 1),
                "decode": round(ab["decode_attn"] / (stage_ms["decode_attn"] * 1e-3) / 1e9, 1)},
        "frac_of_measured_hbm": {"evict": round(ab["evict"] / (evict_us * 1e-6) / 1e9 / peak, 4),
                                 "decode": round(ab["decode_attn"] / (stage_ms["decode_attn"] * 1e-3) / 1e9 / peak, 4),
                                 "step": round(value / world / peak, 4)},
        "frac_of_8tbs": round(value / world / NOMINAL_HBM_GBS, 4),
        "roofline": roof,
        "stage_roofline": sroof,
        "alpha_sweep": sweep,
        "prefill_lse_variant": lse_var,
        "e2e": e2e,
        "gpu_launches": int(launches),
        "gpu_launches_per_step": int(kernels_per_step),
        "clocks": clocks,
    }
    return res


def window_lse_torch(torch, wl, lay, dev):
    """Input preparation for the one-pass variant (plain PyTorch, untimed):
    each window row's natural-log sum of exp over the keys it sees, as a
    causal prefill attention hands it over. [B][Hq][W] float32."""
    B, G, W = len(lay["n"]), wl.group, wl.window
    out = torch.empty((B, wl.hq, W), dtype=torch.float32, device=dev)

    def f32(x):
        if wl.dtype == "bf16":
            return torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).view(torch.bfloat16).to(dev).float()
        return torch.from_numpy(np.ascontiguousarray(x)).to(dev)

    q = f32(lay["q_win"])
    for b in range(B):
        n, off = int(lay["n"][b]), int(lay["kv_offset"][b])
        P = n - W
        mask = torch.arange(n, device=dev)[None, :] > (P + torch.arange(W, device=dev))[:, None]
        for g in range(wl.hkv):
            Kg = f32(lay["K"][g, off:off + n])
            s = torch.matmul(q[b, g * G:(g + 1) * G], Kg.t()) / math.sqrt(wl.head_dim)
            s.masked_fill_(mask[None], float("-inf"))
            out[b, g * G:(g + 1) * G] = torch.logsumexp(s, dim=-1)
            del s, Kg
    return out


def time_lse_variant(torch, tb, dev, stream, wl, lay, desc, layers, stage_ms, step_ms, n, peaks, evict_bytes):
    """tb_window_scores_lse (one QK^T pass, the window rows' normalisers
    given by the prefill) timed on the same rotated layers, and the step it
    gives with the other stages as measured."""
    prev = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = False
    try:
        lse = window_lse_torch(torch, wl, lay, dev)
    finally:
        torch.backends.cuda.matmul.allow_tf32 = prev
    cap = torch.cuda.Stream(dev)
    for d in layers:
        tb.tb_window_scores_lse(desc, d["q_win"], d["K"], lse, d["scores"], d["ews"], stream=stream)
    torch.cuda.synchronize(dev)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=cap):
        for d in layers:
            tb.tb_window_scores_lse(desc, d["q_win"], d["K"], lse, d["scores"], d["ews"], stream=cap)
    with torch.cuda.stream(stream):
        for _ in range(3):
            g.replay()
    torch.cuda.synchronize(dev)
    reps = max(3, 60 // len(layers))
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        t0.record(stream)
        for _ in range(reps):
            g.replay()
        t1.record(stream)
    torch.cuda.synchronize(dev)
    for d in layers:
        st, raw = tb.tb_read_status(d["ews"], stream=stream)
        assert st == tb.TB_OK, raw
    us = 1e3 * t0.elapsed_time(t1) / (reps * len(layers))
    flops = 2.0 * wl.hq * wl.window * wl.head_dim * float(np.sum(n) - len(n) * wl.window)
    tf = flops / (us * 1e-6) / 1e12
    peak = float(peaks["bf16_tflops"])
    # the step with this call in place of tb_window_scores: the measured step
    # time less the difference of the two calls' stage times
    step = 1e3 * (step_ms - stage_ms["window_scores"]) + us
    # the eviction (this call, the select and the gather, each timed alone)
    # against the measured copy bandwidth, as the headline's eviction fraction
    evict_us = us + 1e3 * (stage_ms["select_topk"] + stage_ms["gather_kv"])
    evict_gbs = evict_bytes / (evict_us * 1e-6) / 1e9
    return {"call": "tb_window_scores_lse", "us": round(us, 2),
            "timing": "CUDA graph of one call per rotated layer buffer, events around the replays",
            "flops": flops, "achieved_tflops": round(tf, 1), "tensor_frac": round(tf / peak, 4),
            "step_us_with_it": round(step, 2),
            "evict_us_with_it": round(evict_us, 2), "evict_gbs_with_it": round(evict_gbs, 1),
            "evict_frac_with_it": round(evict_gbs / float(peaks["hbm_gbs"]), 4),
            "note": "one QK^T pass over the prefix keys; the window rows' log-sum-exp comes from the prefill"}


def time_stages(torch, dev, stream, cap, S, K):
    """Per-stage device time per launch: for each stage one CUDA graph of
    that stage's call on every buffer of its rotation in turn (the eviction
    stages over the layer buffers, whose K and V exceed L2 three times; the
    decode over its own rotation of compacted caches, likewise beyond L2),
    replayed with CUDA events around the replays. This is the stage's
    launch duration plus the gap between two kernels of a graph; the step
    graph's own time (the headline) also holds the interaction between
    stages (e.g. the L2 write-back of the gather's output)."""
    out, rot = {}, {}
    for name in STAGES:
        bufs = S["dec_bufs"] if name == "decode_attn" else S["bufs"]
        L = len(bufs)
        reps = max(3, -(-K // L))
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=cap):
            for d in bufs:
                S["stage_call"](name, d, cap)
        with torch.cuda.stream(stream):
            for _ in range(2):
                g.replay()
        torch.cuda.synchronize(dev)
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            t0.record(stream)
            for _ in range(reps):
                g.replay()
            t1.record(stream)
        torch.cuda.synchronize(dev)
        out[name] = t0.elapsed_time(t1) / (reps * L)
        rot[name] = L
        del g
    return out, ("per stage: one CUDA graph of the stage's call on each buffer of its rotation "
                 "(%d layer buffers; the decode over %d compacted caches), replayed between CUDA events"
                 % (rot["window_scores"], rot["decode_attn"]))


def run_e2e(args, wl, tb, torch, dev, stream, lay, desc, ddesc, ews, dws, step_in, ab, R):
    """The same step through the public API from pinned HOST buffers: every
    step copies its inputs host->device and reads its results back. With one
    request the copies are issued per KV head on a copy stream and each
    head's eviction (tb_score_evict on that head's rows) starts once its
    rows have landed, so the evictions overlap the remaining copies; the
    decode follows the last head. The serial form (all copies, then the
    whole eviction) and a copy-only step are timed beside it."""
    steps = args.e2e_steps if args.e2e_steps is not None else min(args.steps, 10)
    if steps <= 0:
        return None
    B = len(lay["n"])
    G = wl.group

    def host(x):
        if wl.dtype == "bf16":
            t = torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).view(torch.bfloat16)
        else:
            t = torch.from_numpy(np.ascontiguousarray(x))
        return t.pin_memory()

    h = {k: host(lay[k]) for k in ("q_win", "K", "V")}
    hq, hk, hv = host(step_in["q"]), host(step_in["k_new"]), host(step_in["v_new"])
    d = {k: torch.empty_like(v, device=dev) for k, v in h.items()}
    qd, kd, vd = torch.empty_like(hq, device=dev), torch.empty_like(hk, device=dev), torch.empty_like(hv, device=dev)
    score_rows, idx_rows = tb.tb_evict_layout(desc)
    idx = torch.empty((wl.hkv, idx_rows), dtype=torch.int32, device=dev)
    Kc = torch.zeros((wl.hkv, desc.out_rows, wl.head_dim), dtype=d["K"].dtype, device=dev)
    Vc = torch.zeros_like(Kc)
    ew = torch.empty(ews, dtype=torch.uint8, device=dev)
    dw = torch.empty(dws, dtype=torch.uint8, device=dev)
    tb.tb_decode_workspace_prepare(ddesc, dw, stream=stream)
    out = torch.empty((B, wl.hq, wl.head_dim), dtype=torch.float32, device=dev)
    lens = torch.tensor([r + 1 for r in R], dtype=torch.int32, device=dev)
    idx_h = torch.empty(idx.shape, dtype=torch.int32).pin_memory()
    out_h = torch.empty(out.shape, dtype=torch.float32).pin_memory()
    rows = [int(desc.out_offset[b]) + R[b] for b in range(B)]
    copy_stream = torch.cuda.Stream(dev)
    per_head = B == 1
    if per_head:   # one KV head's eviction: its G query heads, its K and V rows
        hdesc = tb.EvictDesc(hq=G, hkv=1, head_dim=wl.head_dim, window=wl.window, pool_k=wl.pool_k,
                             dtype=desc.dtype, n=desc.n, alpha=desc.alpha, kv_offset=desc.kv_offset,
                             kv_rows=desc.kv_rows, out_offset=desc.out_offset, out_cap=desc.out_cap,
                             out_rows=desc.out_rows, flags=desc.flags)
        hws = torch.empty(tb.tb_evict_workspace_size(hdesc), dtype=torch.uint8, device=dev)
        landed = [torch.cuda.Event() for _ in range(wl.hkv)]

    def tail():
        qd.copy_(hq, non_blocking=True)
        kd.copy_(hk, non_blocking=True)
        vd.copy_(hv, non_blocking=True)
        for b in range(B):
            Kc[:, rows[b]] = kd[:, b]
            Vc[:, rows[b]] = vd[:, b]
        tb.tb_decode_attn_prepared(ddesc, qd, Kc, Vc, lens, out, dw, stream=stream)
        idx_h.copy_(idx, non_blocking=True)
        out_h.copy_(out, non_blocking=True)

    def serial():
        with torch.cuda.stream(stream):
            for k in d:
                d[k].copy_(h[k], non_blocking=True)
            tb.tb_score_evict(desc, d["q_win"], d["K"], d["V"], idx, Kc, Vc, None, ew, stream=stream)
            tail()

    def overlapped():
        copy_stream.wait_stream(stream)
        with torch.cuda.stream(copy_stream):
            d["q_win"].copy_(h["q_win"], non_blocking=True)
            for g in range(wl.hkv):
                d["K"][g].copy_(h["K"][g], non_blocking=True)
                d["V"][g].copy_(h["V"][g], non_blocking=True)
                landed[g].record(copy_stream)
        with torch.cuda.stream(stream):
            for g in range(wl.hkv):
                stream.wait_event(landed[g])
                tb.tb_score_evict(hdesc, d["q_win"][:, g * G:(g + 1) * G], d["K"][g], d["V"][g], idx[g], Kc[g],
                                  Vc[g], None, hws, stream=stream)
            tail()

    def copy_only():
        with torch.cuda.stream(stream):
            for k in d:
                d[k].copy_(h[k], non_blocking=True)
            qd.copy_(hq, non_blocking=True)
            kd.copy_(hk, non_blocking=True)
            vd.copy_(hv, non_blocking=True)

    def timed(fn):
        # the best of three timed runs of `steps` steps each (host-side
        # hiccups in the pinned copies otherwise show up in single runs)
        for _ in range(2):
            fn()
        torch.cuda.synchronize(dev)
        best = None
        for _ in range(3):
            t0 = torch.cuda.Event(enable_timing=True)
            t1 = torch.cuda.Event(enable_timing=True)
            t0.record(stream)
            for _ in range(steps):
                fn()
            t1.record(stream)
            torch.cuda.synchronize(dev)
            ms = t0.elapsed_time(t1) / steps
            best = ms if best is None else min(best, ms)
        return best

    ms_serial = timed(serial)
    idx_serial = idx_h.clone()
    ms, same_idx = ms_serial, None
    if per_head:
        ms = timed(overlapped)
        st, raw = tb.tb_read_status(hws, stream=stream)
        assert st == tb.TB_OK, raw
        # the share of retained positions the per-head and the batched calls
        # agree on (the scores' float-atomic sums vary in their last bit from
        # run to run, so keys tied with the k-th threshold can swap)
        a, b = idx_h.numpy(), idx_serial.numpy()
        same_idx = round(float(np.mean([np.intersect1d(a[g], b[g]).size / max(1, a.shape[1])
                                        for g in range(a.shape[0])])), 6)
    ms_copy = timed(copy_only)
    h2d = sum(v.numel() * v.element_size() for v in h.values()) + sum(
        v.numel() * v.element_size() for v in (hq, hk, hv))
    d2h = idx_h.numel() * 4 + out_h.numel() * 4
    return {"value": round(ab["step"] / (ms * 1e-3) / 1e9, 1), "unit": "GB/s", "ms_per_step": round(ms, 4),
            "steps": steps, "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "form": ("per-KV-head copies on a copy stream, each head's tb_score_evict after its rows land"
                     if per_head else "all copies, then tb_score_evict and the decode"),
            "serial_ms_per_step": round(ms_serial, 4),
            "copy_only_ms_per_step": round(ms_copy, 4),
            "pinned_h2d_gbs": round(h2d / (ms_copy * 1e-3) / 1e9, 1),
            "copy_bound_frac": round(ms_copy / ms, 4),
            "per_head_idx_agreement_with_batched": same_idx}


def describe(wl, n, a):
    ns = sorted(set(int(x) for x in n))
    nd = ("N=%d" % ns[0]) if len(ns) == 1 else ("N in [%d, %d] (%d requests)" % (min(ns), max(ns), len(n)))
    return "%s: %dq/%dkv heads, d=%d, %s, batch %d, %s, W=%d, pool %d" % (
        wl.name, wl.hq, wl.hkv, wl.head_dim, wl.dtype, len(n), nd, wl.window, wl.pool_k)


# ---------------------------------------------------------------------------
# CPU oracle (cpu_baseline leg and the reference arm)
# ---------------------------------------------------------------------------

def oracle_sample(wl, lay, heads, n_keys=None):
    """Times the oracle on KV heads `heads` of request 0 (optionally on the
    first n_keys prompt tokens only); returns (seconds, algorithmic bytes)."""
    from oracle import timebill_oracle as orc
    q = inputs.as_f32(lay["q_win"], wl.dtype)
    K = inputs.as_f32(lay["K"], wl.dtype)
    V = inputs.as_f32(lay["V"], wl.dtype)
    n = int(lay["n"][0]) if n_keys is None else int(n_keys)
    a = float(lay["alpha"][0])
    G = wl.group
    off = int(lay["kv_offset"][0])
    e = elem_bytes(wl)
    row = e * wl.head_dim
    t0 = time.perf_counter()
    byt = 0
    for g in heads:
        res = orc.score_evict(q[:1, g * G:(g + 1) * G], K[g:g + 1, off:off + n], V[g:g + 1, off:off + n],
                              [n], [a], [0], wl.window, wl.pool_k)[0]
        R = res["R"]
        Kc = np.concatenate([res["Kc"][0], K[g, off + n - 1:off + n]])
        Vc = np.concatenate([res["Vc"][0], V[g, off + n - 1:off + n]])
        qd = q[0, g * G:(g + 1) * G, 0]
        orc.decode_attention(qd, Kc[None], Vc[None], R + 1)
        byt += row * (n + 4 * R) + G * wl.window * wl.head_dim * e + 2 * row * (R + 1)
    return time.perf_counter() - t0, byt


def cpu_baseline(args, wl, alpha):
    lay = inputs.make_layer(wl, 0, alpha=alpha)
    heads, secs, byt = [], 0.0, 0
    for g in range(wl.hkv):
        s, b = oracle_sample(wl, lay, [g])
        heads.append(g)
        secs += s
        byt += b
        if secs >= args.cpu_seconds:
            break
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    return {"value": round(byt / secs / 1e9, 4), "unit": "GB/s", "cores": cores, "kind": "oracle",
            "seconds": round(secs, 2),
            "sample": "eviction of %d of %d KV heads of request 0 of one layer plus one decode step "
                      "over each head's retained cache, numpy fp64" % (len(heads), wl.hkv)}


def run_reference(args, wl, alpha):
    lay = inputs.make_layer(wl, 0, alpha=alpha)
    n_full = int(lay["n"][0])
    # size the per-step sample so that warm-up + steps stay within ~150 s
    s1, _ = oracle_sample(wl, lay, [0], n_keys=min(n_full, 4096))
    per_key = s1 / min(n_full, 4096)
    budget = 150.0 / max(1, args.steps + args.warmup)
    n_keys = int(min(n_full, max(4 * wl.window, budget / max(per_key, 1e-12))))
    for i in range(args.warmup):
        oracle_sample(wl, lay, [i % wl.hkv], n_keys=n_keys)
    secs, byt = 0.0, 0
    for i in range(args.steps):
        s, b = oracle_sample(wl, lay, [i % wl.hkv], n_keys=n_keys)
        secs += s
        byt += b
    value = byt / secs / 1e9
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    sample = ("per step: eviction of one KV head of request 0 over the first %d of %d prompt tokens "
              "plus one decode step, numpy fp64" % (n_keys, n_full))
    return {
        "impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": "GB/s", "n_gpus": 0,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(1e3 * secs / args.steps, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded Gaussian q/K/V with planted heavy hitters)",
        "config": {"workload": describe(wl, lay["n"], lay["alpha"]), "alpha": float(lay["alpha"][0])},
        "cpu_baseline": {"value": round(value, 4), "unit": "GB/s", "cores": cores, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


# ---------------------------------------------------------------------------
# profiling-based fit of the time model (Eq. 6a / 6b) on these kernels
# ---------------------------------------------------------------------------

def _time_per_call(torch, dev, stream, calls, reps):
    """Device µs per call of `calls` (a list of zero-argument launches on
    `stream`), captured into one CUDA graph and replayed `reps` times."""
    cap = torch.cuda.Stream(dev)
    for c in calls:
        c(stream)
    torch.cuda.synchronize(dev)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=cap):
        for c in calls:
            c(cap)
    with torch.cuda.stream(stream):
        for _ in range(3):
            g.replay()
    torch.cuda.synchronize(dev)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        t0.record(stream)
        for _ in range(reps):
            g.replay()
        t1.record(stream)
    torch.cuda.synchronize(dev)
    return 1e3 * t0.elapsed_time(t1) / (reps * len(calls))


def _fit_report(tb, x, t_us, degree):
    coef, mape = tb.tb_fit_time_model(x, t_us, degree)
    # hold-out: fit on the even-indexed points, score the odd-indexed ones
    ce, _ = tb.tb_fit_time_model(x[0::2], t_us[0::2], degree)
    xo, to = np.asarray(x[1::2], np.float64), np.asarray(t_us[1::2], np.float64)
    hold = 100.0 * float(np.mean(np.abs(np.polyval(ce, xo) - to) / to))
    names = ["p_us_per_token", "q_us"] if degree == 1 else ["a_us_per_token2", "b_us_per_token", "c_us"]
    rep = {k: float("%.6g" % v) for k, v in zip(names, coef)}
    rep.update({"mape_pct": round(mape, 3), "holdout_mape_pct": round(hold, 3),
                "points": [[int(a), round(b, 3)] for a, b in zip(x, t_us)]})
    return rep


def run_time_fit(args):
    """Section "Profiling-based Fitting": measure the path's kernels over a
    range of lengths on the paper's model shape (28 query / 4 KV heads,
    d 128, bf16) and fit Eq. 6b to the decode attention (N_kv in 1K..32K,
    the paper's profiling range) and Eq. 6a's quadratic to the eviction
    (N_x in 2K..32K, alpha 0.5). Every point rotates over enough layer
    buffers that a graph replay reads more than L2 holds."""
    import torch
    from paper_2512_21859_gb300 import binding as tb

    tb.load()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream(dev)
    wl = inputs.WORKLOADS["7b"]
    d, e = wl.head_dim, 2
    gen = torch.Generator(device=dev)
    gen.manual_seed(wl.seed * 1000 + 6)
    sampler = ClockSampler(0)

    dec_x, dec_t = [], []
    for n in range(1024, 32768 + 1, 1024):
        per = 2 * wl.hkv * n * d * e
        L = int(min(256, max(2, math.ceil(3 * L2_BYTES / per))))
        ddesc = tb.DecodeDesc(hq=wl.hq, hkv=wl.hkv, head_dim=d, dtype=tb.TB_BF16, cache_offset=[0],
                              cache_cap=[n], cache_rows=n, max_len=n)
        dws = tb.tb_decode_workspace_size(ddesc)
        kv = torch.randn((L, 2, wl.hkv, n, d), generator=gen, device=dev, dtype=torch.bfloat16)
        q = torch.randn((L, 1, wl.hq, d), generator=gen, device=dev, dtype=torch.bfloat16)
        lens = torch.full((1,), n, dtype=torch.int32, device=dev)
        out = torch.empty((L, 1, wl.hq, d), dtype=torch.float32, device=dev)
        ws = torch.empty((L, max(dws, 1)), dtype=torch.uint8, device=dev)
        for l in range(L):
            tb.tb_decode_workspace_prepare(ddesc, ws[l], stream=stream)
        calls = [lambda st, l=l: tb.tb_decode_attn_prepared(ddesc, q[l], kv[l, 0], kv[l, 1], lens, out[l],
                                                            ws[l], stream=st) for l in range(L)]
        dec_x.append(n)
        dec_t.append(_time_per_call(torch, dev, stream, calls, max(3, 2000 // L)))
        for l in range(L):
            st, raw = tb.tb_read_status(ws[l], stream=stream)
            assert st == tb.TB_OK, raw
        del kv, q, out, ws

    ev_x, ev_t = [], []
    alpha = 0.5
    for n in range(2048, 32768 + 1, 2048):
        lay = inputs.make_layer(wl, 0, alpha=alpha, n_override=[n])
        per = 2 * wl.hkv * n * d * e
        L = int(min(64, max(2, math.ceil(3 * L2_BYTES / per))))
        desc = tb.EvictDesc(hq=wl.hq, hkv=wl.hkv, head_dim=d, window=wl.window, pool_k=wl.pool_k,
                            dtype=tb.TB_BF16, n=lay["n"], alpha=lay["alpha"], kv_offset=lay["kv_offset"],
                            kv_rows=n, out_cap=[retained(n, wl.window, alpha)[1]])
        _, idx_rows = tb.tb_evict_layout(desc)
        ews = tb.tb_evict_workspace_size(desc)

        def dev_bf16(x):
            return torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).view(torch.bfloat16).to(dev)

        base = {k: dev_bf16(lay[k]) for k in ("q_win", "K", "V")}
        bufs = []
        for l in range(L):
            b = {k: (v if l == 0 else v.clone()) for k, v in base.items()}
            b["Kc"] = torch.empty((wl.hkv, desc.out_rows, d), dtype=torch.bfloat16, device=dev)
            b["Vc"] = torch.empty_like(b["Kc"])
            b["idx"] = torch.empty((wl.hkv, idx_rows), dtype=torch.int32, device=dev)
            b["ws"] = torch.empty(ews, dtype=torch.uint8, device=dev)
            bufs.append(b)
        calls = [lambda st, b=b: tb.tb_score_evict(desc, b["q_win"], b["K"], b["V"], b["idx"], b["Kc"],
                                                   b["Vc"], None, b["ws"], stream=st) for b in bufs]
        ev_x.append(n)
        ev_t.append(_time_per_call(torch, dev, stream, calls, max(3, 400 // L)))
        for b in bufs:
            st, raw = tb.tb_read_status(b["ws"], stream=stream)
            assert st == tb.TB_OK, raw
        del bufs, base
    clocks = sampler.stop()
    return {
        "metric": "time-model fit (Eq. 6a / 6b by least squares) of the path's kernels, MAPE %",
        "unit": "us", "data": "synthetic (seeded Gaussian; eviction inputs with planted heavy hitters)",
        "config": {"workload": "7b shape: 28q/4kv heads, d=128, bf16, batch 1, W=32, pool 7",
                   "timing": "CUDA graph of one call per rotated layer buffer (inputs larger than L2), "
                             "CUDA events around the replays"},
        "decode_attn_eq6b": _fit_report(tb, dec_x, dec_t, 1),
        "score_evict_eq6a": dict(_fit_report(tb, ev_x, ev_t, 2), alpha=alpha),
        "clocks": clocks,
    }


def main(argv=None):
    args = parse_args(argv)
    world, rank, local = dist_env()
    wl = inputs.WORKLOADS[args.workload]
    if args.impl == "reference":
        if rank != 0:
            return 0
        print(json.dumps(run_reference(args, wl, args.alpha)), flush=True)
        return 0

    import torch
    if not torch.cuda.is_available():
        print(json.dumps({"error": "no CUDA device: the benchmark times the GPU path only"}))
        return 1
    if args.fit_time_model:
        if rank == 0:
            print(json.dumps(run_time_fit(args)), flush=True)
        return 0
    dist = dist_init(world, True)
    alphas = [float(x) for x in args.sweep.split(",")] if args.sweep else [args.alpha]
    if args.sweep:   # one line per alpha already: no per-alpha table inside each
        args.no_alpha_sweep = True
    base_cpu = None
    for alpha in alphas:
        res = run_ours(args, wl, alpha, world, rank, local, dist)
        if rank == 0:
            if world == 1 and not args.no_cpu_baseline:
                if base_cpu is None or args.sweep:
                    base_cpu = cpu_baseline(args, wl, alpha)
                res["cpu_baseline"] = base_cpu
            print(json.dumps(res), flush=True)
    if dist:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
