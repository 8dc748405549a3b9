"""CPU fp64 oracle for TimeBill's KV-eviction + decode-attention path.

TEST INFRASTRUCTURE ONLY. Nothing in the product path (the CUDA library and
its Python binding) may import or call this module; only the tests, the
smoke check and the benchmark's CPU-baseline leg do. It shares no code with
the CUDA path: it receives plain float arrays and writes its own arithmetic.

What it computes, step by step, for each request and KV head (all in fp64
from the exact input values):

1. Budget (Eq. 8, Section "End-to-end Execution Time Prediction"): after
   evicting a fraction alpha of the N prompt tokens, k = ceil((1-alpha) N)
   prefix tokens are retained on top of the W observation-window tokens,
   clamped to the P = N - W prefix tokens available.
2. Window logits (attention definition, Section "FLOPs-based Modeling"):
   s = q . k / sqrt(d) for every window query q of every query head of the
   group and every key it may see (window row w sees keys j <= P + w).
3. Row softmax over the visible keys, then the score of prefix key j is the
   sum of its probabilities over the window rows and the group's query heads
   (SnapKV-style observation-window voting; the paper names SnapKV as its
   eviction method in "Experimental Setup"). The same sums from given row
   log-sum-exp values (a prefill attention's normalisers) are
   window_scores_from_lse; window_lse computes those normalisers.
4. 1-D max-pool of the scores with an odd kernel, stride 1, same padding
   (out-of-range neighbours ignored).
5. The k prefix positions with the largest pooled score, ties to the lower
   index, plus every window position, in ascending order.
6. The compact cache: bit copies of those K and V rows.
7. Decode-step attention (Eq. 8's N_kv^i keys, attention definition): one
   query per head over the first ``len`` rows of the compact cache.
8. The eviction ratio the time budget allows (Prob. 13 of "Time-Budgeted LLM
   Inference Mechanism"): the smallest alpha in [0, alpha_max] whose
   worst-case execution time estimate (Eq. 12, built from Eqs. 6a, 9-11)
   fits the budget, found here from its definition by bisection.
9. Profiling-based fitting (Section "Profiling-based Fitting"): the
   least-squares coefficients of Eq. 6a (degree 2) or Eq. 6b (degree 1)
   through measured (length, time) pairs, and the fit's mean absolute
   percentage error (the accuracy measure of the time-model evaluation).

Parity status: every function here is pinned by tests/test_oracle_pins.py
(hand-derived closed forms, brute force, invariants, library routines).
"""
from __future__ import annotations

import math
from typing import List, Optional, Sequence, Tuple

import numpy as np

__all__ = [
    "retained_count",
    "window_scores",
    "window_lse",
    "window_scores_from_lse",
    "max_pool",
    "avg_pool",
    "select_indices",
    "gather_rows",
    "score_evict",
    "decode_attention",
    "decode_batch",
    "pessimistic_length",
    "wcet",
    "alpha_star",
    "fit_time_model",
]


def retained_count(n: int, window: int, alpha: float,
                   budget_includes_window: bool = False) -> Tuple[int, int]:
    """(k, R): retained prefix tokens and retained rows per KV head.

    Eq. 8 gives the cache length after evicting a fraction alpha of the N
    prompt tokens as (1-alpha) N. Reading: the observation window is kept on
    top of ceil((1-alpha) N) prefix tokens, clamped to the P = N - W prefix
    tokens (so alpha = 0 keeps the whole prompt). The ceiling is taken of
    (1-alpha) N - 1e-9 N so that a decimal alpha whose binary value lands a
    hair above an integer product (alpha=0.3, N=10) rounds as written.
    With budget_includes_window, Eq. 8 is read literally instead: the whole
    retained cache, window included, is the ceil((1-alpha) N) rows, so the
    prefix gets that count less W (still clamped; the window stays).
    """
    n = int(n)
    window = int(window)
    if window < 1 or window > n:
        raise ValueError("need 1 <= window <= n")
    if not (0.0 <= alpha <= 1.0):
        raise ValueError("alpha must lie in [0, 1]")
    p = n - window
    k = math.ceil((1.0 - alpha) * n - 1e-9 * n)
    if budget_includes_window:
        k -= window
    k = min(max(k, 0), p)
    return k, k + window


def window_scores(q_win: np.ndarray, K: np.ndarray) -> np.ndarray:
    """Observation-window scores S[g, j] for the prefix keys of one request.

    q_win: [Hq][W][d] window queries; K: [Hkv][N][d] keys. Query head h
    belongs to KV head g = h // (Hq / Hkv). Returns S: [Hkv][P] (fp64).
    """
    q = np.asarray(q_win, dtype=np.float64)
    k = np.asarray(K, dtype=np.float64)
    hq, W, d = q.shape
    hkv, N, _ = k.shape
    G = hq // hkv
    P = N - W
    sigma = 1.0 / math.sqrt(d)
    # visible[w, j]: window row w (absolute position P + w) sees keys j <= P + w
    visible = np.arange(N)[None, :] <= (P + np.arange(W))[:, None]
    S = np.zeros((hkv, P), dtype=np.float64)
    for g in range(hkv):
        for h in range(g * G, (g + 1) * G):
            logits = sigma * (q[h] @ k[g].T)            # [W][N]
            logits = np.where(visible, logits, -np.inf)
            m = logits.max(axis=1, keepdims=True)
            e = np.exp(logits - m)
            prob = e / e.sum(axis=1, keepdims=True)
            S[g] += prob[:, :P].sum(axis=0)
    return S


def window_lse(q_win: np.ndarray, K: np.ndarray) -> np.ndarray:
    """Log-sum-exp of every window row's logits over the keys it sees: the
    softmax normaliser of the attention definition, log sum_j exp(s_j), for
    row w of head h over keys j <= P + w (what a causal prefill attention
    produces for the last W query rows). Returns [Hq][W] (fp64)."""
    q = np.asarray(q_win, dtype=np.float64)
    k = np.asarray(K, dtype=np.float64)
    hq, W, d = q.shape
    hkv, N, _ = k.shape
    G = hq // hkv
    P = N - W
    sigma = 1.0 / math.sqrt(d)
    # row w's last visible key is its own position P + w
    last_seen = P + np.arange(W)
    visible = np.arange(N)[None, :] <= last_seen[:, None]
    out = np.zeros((hq, W), dtype=np.float64)
    for h in range(hq):
        logits = np.where(visible, sigma * (q[h] @ k[h // G].T), -np.inf)
        m = logits.max(axis=1)
        out[h] = m + np.log(np.exp(logits - m[:, None]).sum(axis=1))
    return out


def window_scores_from_lse(q_win: np.ndarray, K: np.ndarray, lse: np.ndarray) -> np.ndarray:
    """Step 3 with the row normalisers given: S[g, j] = sum over the heads h
    of group g and window rows w of exp(s_hwj - lse[h, w]), prefix keys
    j < P (all of them visible to every window row). Returns [Hkv][P]."""
    q = np.asarray(q_win, dtype=np.float64)
    k = np.asarray(K, dtype=np.float64)
    L = np.asarray(lse, dtype=np.float64)
    hq, W, d = q.shape
    hkv, N, _ = k.shape
    G = hq // hkv
    P = N - W
    sigma = 1.0 / math.sqrt(d)
    S = np.zeros((hkv, P), dtype=np.float64)
    for h in range(hq):
        logits = sigma * (q[h] @ k[h // G, :P].T)      # [W][P]
        S[h // G] += np.exp(logits - L[h][:, None]).sum(axis=0)
    return S


def max_pool(S: np.ndarray, pool_k: int) -> np.ndarray:
    """1-D max-pool along the last axis: kernel pool_k (odd), stride 1, same
    padding with out-of-range positions ignored."""
    if pool_k < 1 or pool_k % 2 == 0:
        raise ValueError("pool_k must be odd and >= 1")
    S = np.asarray(S, dtype=np.float64)
    out = S.copy()
    L = S.shape[-1]
    for t in range(1, pool_k // 2 + 1):
        if t >= L:
            break
        out[..., t:] = np.maximum(out[..., t:], S[..., :-t])   # neighbour on the left
        out[..., :-t] = np.maximum(out[..., :-t], S[..., t:])  # neighbour on the right
    return out


def avg_pool(S: np.ndarray, pool_k: int) -> np.ndarray:
    """1-D average pool along the last axis (SnapKV's pooling): kernel pool_k
    (odd), stride 1, same padding with zeros, so every output is the sum of
    the in-range neighbours divided by pool_k."""
    if pool_k < 1 or pool_k % 2 == 0:
        raise ValueError("pool_k must be odd and >= 1")
    S = np.asarray(S, dtype=np.float64)
    half = pool_k // 2
    L = S.shape[-1]
    pad = np.zeros(S.shape[:-1] + (half,))
    Z = np.concatenate([pad, S, pad], axis=-1)
    total = np.zeros_like(S)
    for t in range(pool_k):
        total += Z[..., t:t + L]
    return total / pool_k


def select_indices(pooled: np.ndarray, k: int, n: int) -> np.ndarray:
    """Retained positions of one KV head: the k prefix positions with the
    largest pooled score (ties to the lower index), then the window
    positions P..n-1; ascending int64."""
    pooled = np.asarray(pooled, dtype=np.float64)
    P = pooled.shape[0]
    order = np.lexsort((np.arange(P), -pooled))   # score descending, index ascending
    keep = np.sort(order[:k])
    return np.concatenate([keep, np.arange(P, n)]).astype(np.int64)


def gather_rows(X: np.ndarray, idx: np.ndarray) -> np.ndarray:
    """Rows idx of X (a bit copy)."""
    return np.asarray(X)[np.asarray(idx, dtype=np.int64)]


def score_evict(q_win: np.ndarray, K: np.ndarray, V: np.ndarray, n: Sequence[int],
                alpha: Sequence[float], kv_offset: Sequence[int], window: int,
                pool_k: int, heads: Optional[Sequence[int]] = None, pool: str = "max",
                budget_includes_window: bool = False) -> List[dict]:
    """The whole eviction for a packed batch.

    q_win [B][Hq][W][d]; K, V [Hkv][rows][d] with request b at rows
    kv_offset[b] .. kv_offset[b] + n[b]. Returns, per request, a dict with
    k, R, S [Hkv][P], pooled [Hkv][P], idx [Hkv][R], Kc/Vc [Hkv][R][d]
    (in the input array's dtype). ``heads`` restricts the work to some KV
    heads (the other rows stay zero / empty). ``pool`` is "max" (the
    default reading) or "avg"; ``budget_includes_window`` selects the literal
    reading of Eq. 8 in retained_count.
    """
    if pool not in ("max", "avg"):
        raise ValueError("pool must be 'max' or 'avg'")
    out = []
    hkv = K.shape[0]
    G = q_win.shape[1] // hkv
    for b in range(len(n)):
        nb, off = int(n[b]), int(kv_offset[b])
        k, R = retained_count(nb, window, float(alpha[b]), budget_includes_window)
        P = nb - window
        hs = range(hkv) if heads is None else heads
        S = np.zeros((hkv, P))
        pooled = np.zeros((hkv, P))
        idx = np.zeros((hkv, R), dtype=np.int64)
        Kc = np.zeros((hkv, R, K.shape[2]), dtype=K.dtype)
        Vc = np.zeros_like(Kc)
        for g in hs:
            Kg = K[g:g + 1, off:off + nb]
            S[g] = window_scores(q_win[b, g * G:(g + 1) * G], Kg)[0]
            pooled[g] = max_pool(S[g], pool_k) if pool == "max" else avg_pool(S[g], pool_k)
            idx[g] = select_indices(pooled[g], k, nb)
            Kc[g] = gather_rows(K[g, off:off + nb], idx[g])
            Vc[g] = gather_rows(V[g, off:off + nb], idx[g])
        out.append({"k": k, "R": R, "S": S, "pooled": pooled, "idx": idx,
                    "Kc": Kc, "Vc": Vc})
    return out


def decode_attention(q: np.ndarray, Kc: np.ndarray, Vc: np.ndarray, length: int) -> np.ndarray:
    """One decode step for one request: q [Hq][d]; Kc, Vc [Hkv][>=length][d].
    Returns [Hq][d] fp64: softmax(q . k / sqrt(d)) weighted sum of v over the
    first ``length`` cache rows of the head's KV group."""
    q = np.asarray(q, dtype=np.float64)
    hq, d = q.shape
    hkv = Kc.shape[0]
    G = hq // hkv
    sigma = 1.0 / math.sqrt(d)
    out = np.zeros((hq, d), dtype=np.float64)
    if length <= 0:
        return out
    for h in range(hq):
        g = h // G
        kk = np.asarray(Kc[g, :length], dtype=np.float64)
        vv = np.asarray(Vc[g, :length], dtype=np.float64)
        s = sigma * (kk @ q[h])
        e = np.exp(s - s.max())
        out[h] = (e / e.sum()) @ vv
    return out


def decode_batch(q: np.ndarray, Kc: np.ndarray, Vc: np.ndarray, lens: Sequence[int],
                 cache_offset: Sequence[int]) -> np.ndarray:
    """Decode step for a packed batch: q [B][Hq][d]; Kc, Vc [Hkv][rows][d]
    with request b's cache at rows cache_offset[b] ..; returns [B][Hq][d]."""
    B = q.shape[0]
    out = np.zeros(q.shape, dtype=np.float64)
    for b in range(B):
        off, L = int(cache_offset[b]), int(lens[b])
        out[b] = decode_attention(q[b], Kc[:, off:off + L], Vc[:, off:off + L], L)
    return out


# ---------------------------------------------------------------------------
# step 8: the eviction ratio a time budget allows
# ---------------------------------------------------------------------------

def pessimistic_length(n_hat: float, k: float, n_max: int) -> int:
    """N_W = min(k N_hat, N_max) (Section "End-to-end Execution Time
    Prediction"). Reading: k N_hat is rounded up, the pessimistic side, since
    it counts decoding steps."""
    return int(min(math.ceil(k * n_hat), n_max))


def wcet(a: float, b: float, c: float, p: float, q: float, n_x: int, alpha: float,
         n_w: int) -> float:
    """Eq. 12: the prefill time of Eq. 6a plus the decoding phase of Eq. 11,
    the sum over steps i = 1 .. N_W - 1 of Eq. 10, p ((1 - alpha) N_x + i - 1) + q.
    The sum is taken term by term."""
    t_prefill = a * n_x * n_x + b * n_x + c
    t_decode = 0.0
    for i in range(1, n_w):
        t_decode += p * ((1.0 - alpha) * n_x + i - 1) + q
    return t_prefill + t_decode


def alpha_star(a: float, b: float, c: float, p: float, q: float, n_x: int, n_hat: float,
               k: float, n_max: int, t_predict: float, budget: float,
               alpha_max: float) -> float:
    """Prob. 13: minimise alpha subject to t_Predict + WCET(alpha) <= T and
    0 <= alpha <= alpha_max. WCET is non-increasing in alpha (p > 0), so the
    smallest feasible alpha is found by bisection on the constraint itself.
    When no alpha in range meets the budget, alpha_max (the most the budget
    can be helped; the paper's overrun strategies take it from there)."""
    n_w = pessimistic_length(n_hat, k, n_max)

    def excess(al: float) -> float:
        return t_predict + wcet(a, b, c, p, q, n_x, al, n_w) - budget

    if excess(0.0) <= 0.0:
        return 0.0
    if excess(alpha_max) > 0.0:
        return float(alpha_max)
    lo, hi = 0.0, float(alpha_max)  # excess(lo) > 0 >= excess(hi)
    for _ in range(80):
        mid = 0.5 * (lo + hi)
        if excess(mid) <= 0.0:
            hi = mid
        else:
            lo = mid
    return hi


# ---------------------------------------------------------------------------
# step 9: profiling-based fitting of the time model
# ---------------------------------------------------------------------------

def fit_time_model(x: Sequence[float], t: Sequence[float], degree: int) -> Tuple[List[float], float]:
    """Least squares (the fitting method the paper names) of t ~ poly(x) with
    the form of Eq. 6a (degree 2: a x^2 + b x + c) or Eq. 6b (degree 1:
    p x + q). Returns the coefficients, highest power first, and the MAPE in
    percent over the same points: 100/n sum |poly(x_i) - t_i| / t_i.
    The least-squares solve is numpy's lstsq on the Vandermonde matrix."""
    xa = np.asarray(x, dtype=np.float64)
    ta = np.asarray(t, dtype=np.float64)
    V = np.stack([xa ** k for k in range(degree, -1, -1)], axis=1)
    coef = np.linalg.lstsq(V, ta, rcond=None)[0]
    fit = V @ coef
    mape = 100.0 * float(np.mean(np.abs(fit - ta) / ta))
    return [float(c) for c in coef], mape
