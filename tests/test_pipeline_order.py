"""The pipelined layer loop's ordering, checked on a model of its launches.

The bench replays pipelined_step (bench.py) from CUDA graphs. Each stage's
kernel is chained to the one before it by programmatic dependent launch.
This test rebuilds the happens-before graph that this chaining gives, from
each kernel's documented behaviour (include/timebill_kv.h and the kernels'
sources):
- launch: a kernel starts once the kernel before it lets its dependents
  start; the first kernel of a graph launch starts once the previous graph
  launch has completed;
- wait: a kernel that waits before its work begins that work only once the
  kernel before it has completed, and a kernel without that wait begins at
  once;
- trigger: the point where a kernel lets its dependents start, right after
  its wait, at its start, or at its exit;
- end wait: a concurrent decode or gather (TB_DECODE_CONCURRENT,
  TB_EVICT_GATHER_CONCURRENT) completes only after the kernel before it.
For every two calls that touch the same buffer, at least one of them writing
it, the test checks that the earlier call's completion happens before the
later call's first access, across several replays of the rotation graph and
the one-step graphs after them. The negative control leaves out the end wait
and finds two unordered pairs. One is the gather's read of indices that no
wait orders after their select. The other is its overwrite of a compacted
cache that no wait orders after the decode that read it.
"""
import collections
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402

# kernel: (waits before its work, trigger point, waits at its end, reads, writes)
# buffers are per layer: K, V, q_win (inputs), ews (eviction workspace:
# control words and status), scores, idx, Kc (compacted K and V), out and
# sdws (the step decode's output and workspace)
KERNELS = {
    "window_scores": [  # the clearing kernel, then the fused two-pass scoring
        ("clear_words", True, "after_wait", False, [], ["ews"]),
        ("ws_tc", True, "exit", False, ["K", "q_win", "ews"], ["scores", "ews"]),
    ],
    "select_topk": [("select_cluster", True, "after_wait", False, ["scores"], ["idx", "ews"])],
    "decode_beside_select": [("decode_tma", False, "start", True, ["Kc", "sdws"], ["out", "sdws"])],
    "gather_beside_select": [("gather", False, "start", True, ["idx", "K", "V"], ["Kc"])],
    # without the concurrent flag: the gather waits for the kernel before it
    "gather_kv": [("gather", True, "after_wait", False, ["idx", "K", "V"], ["Kc"])],
    # tb_score_evict: its clearing kernel, the scoring, the select, then its
    # own gather (which never takes the concurrent flag)
    "score_evict": [
        ("clear_words", True, "after_wait", False, [], ["ews"]),
        ("ws_tc", True, "exit", False, ["K", "q_win", "ews"], ["scores", "ews"]),
        ("select_cluster", True, "after_wait", False, ["scores"], ["idx", "ews"]),
        ("gather", True, "after_wait", False, ["idx", "K", "V"], ["Kc"]),
    ],
}


def _program(L, replays, tail):
    """Graph launches in order, each a list of (call, buffer)."""
    rotation = [c for i in range(L) for c in bench.pipelined_step(i, L)]
    return [rotation] * replays + [bench.pipelined_step(i, L) for i in range(tail)]


def _build(program, end_wait=True):
    """Kernel instances and the happens-before edges between their events
    (start, wait return, first access, trigger, completion)."""
    ks, edges = [], collections.defaultdict(set)
    prev_launch = []
    for launch in program:
        this_launch, prev = [], None
        for call, buf in launch:
            for name, waits, trig, endw, reads, writes in KERNELS[call]:
                k = len(ks)
                ks.append(dict(name=name, call=call, buf=buf, reads=reads, writes=writes))
                S, W, R, T, C = (k, "start"), (k, "wait"), (k, "access"), (k, "trigger"), (k, "done")
                if prev is None:
                    for p in prev_launch:  # a graph launch starts after the previous one completed
                        edges[(p, "done")].add(S)
                else:
                    edges[(prev, "trigger")].add(S)
                edges[S].add(W)
                if waits and prev is not None:
                    edges[(prev, "done")].add(W)
                edges[W if waits else S].add(R)
                if trig == "exit":
                    edges[C].add(T)
                else:
                    edges[W if trig == "after_wait" else S].add(T)
                    edges[T].add(C)
                edges[R].add(C)
                if endw and end_wait and prev is not None:
                    edges[(prev, "done")].add(C)
                this_launch.append(k)
                prev = k
        prev_launch = this_launch
    return ks, edges


def _reach(edges, src):
    seen, todo = {src}, [src]
    while todo:
        for v in edges.get(todo.pop(), ()):
            if v not in seen:
                seen.add(v)
                todo.append(v)
    return seen


def _unordered(ks, edges):
    """Pairs of kernels touching one buffer (one of them writing it) where the
    earlier one's completion does not happen before the later one's access."""
    bad = []
    reach = {}
    for b in range(len(ks)):
        kb = ks[b]
        for a in range(b):
            ka = ks[a]
            if ka["buf"] != kb["buf"]:
                continue
            shared = [x for x in set(ka["reads"] + ka["writes"]) & set(kb["reads"] + kb["writes"])
                      if x in ka["writes"] or x in kb["writes"]]
            if not shared:
                continue
            if a not in reach:
                reach[a] = _reach(edges, (a, "done"))
            if (b, "access") not in reach[a]:
                bad.append((ka["name"], kb["name"], ka["buf"], shared))
    return bad


@pytest.mark.parametrize("L", [2, 3, 4])
def test_every_hazard_is_ordered(L):
    ks, edges = _build(_program(L, replays=3, tail=L - 1))
    assert len(ks) == (3 * L + L - 1) * 5
    assert _unordered(ks, edges) == []


@pytest.mark.parametrize("L", [2, 3])
def test_without_the_end_wait_two_hazards_are_unordered(L):
    """The gather's read of the indices its select wrote a step earlier, and
    its overwrite of a compacted cache that a decode read before: nothing
    but the end waits orders either."""
    ks, edges = _build(_program(L, replays=3, tail=0), end_wait=False)
    kinds = {(a, b, tuple(sh)) for a, b, _, sh in _unordered(ks, edges)}
    assert kinds == {("select_cluster", "gather", ("idx",)), ("decode_tma", "gather", ("Kc",))}


def test_the_schedule_touches_distinct_buffers_within_a_step():
    """Within one step the decode's cache, the gather's layer and the scored
    layer are three different buffers for L >= 3, and the decode and the
    gather differ for L = 2."""
    for L in (2, 3, 4, 6):
        for i in range(2 * L):
            calls = dict(bench.pipelined_step(i, L))
            assert calls["window_scores"] == calls["select_topk"] == i % L
            assert calls["decode_beside_select"] != calls["gather_beside_select"]
            if L >= 3:
                assert len({calls["window_scores"], calls["decode_beside_select"],
                            calls["gather_beside_select"]}) == 3


@pytest.mark.parametrize("end_wait", [True, False])
def test_the_gather_after_a_concurrent_decode_on_the_same_stream(end_wait):
    """One layer's scores and select, the concurrent decode over another
    layer's cache, then the plain gather of the select's rows on the same
    stream (no event): the gather waits for the decode only, so its read of
    the indices is ordered after the select exactly when the decode's grid
    completes after the select. Without that, nothing later on the stream is
    ordered after the select: the next call's clearing kernel, scoring and
    select on that layer are not either."""
    launch = [("window_scores", 0), ("select_topk", 0), ("decode_beside_select", 1), ("gather_kv", 0)]
    ks, edges = _build([launch * 3], end_wait=end_wait)  # eager: one chain, no graph boundaries
    bad = {(a, b) for a, b, _, _ in _unordered(ks, edges)}
    if end_wait:
        assert bad == set()
    else:
        assert {a for a, _ in bad} == {"select_cluster"}
        assert ("select_cluster", "gather") in bad


def test_score_evict_calls_in_a_row():
    """tb_score_evict on one workspace and layer, call after call, eagerly
    (every call its own launch sequence on one stream, PDL-chained)."""
    ks, edges = _build([[("score_evict", 0)] * 4])
    assert _unordered(ks, edges) == []
