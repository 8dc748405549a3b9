"""Independent pure-Python restatement of the eviction rule for tiny inputs.

Element-by-element loops with the math module only (no numpy), written
separately from the oracle so that the two can pin each other: window
logits q.k/sqrt(d) with the causal window mask, per-row softmax, the sum
over window rows and group heads, a max-pool over explicit neighbour lists,
and a full comparison sort (score descending, index ascending).
"""
import math


def budget(n, window, alpha):
    k = math.ceil((1.0 - alpha) * n - 1e-9 * n)
    return max(0, min(k, n - window))


def scores(q_win, K, group):
    """q_win[h][w][i], K[g][j][i] as nested lists; returns S[g][j] for j < P."""
    hq = len(q_win)
    W = len(q_win[0])
    d = len(q_win[0][0])
    hkv = len(K)
    N = len(K[0])
    P = N - W
    S = [[0.0] * P for _ in range(hkv)]
    for h in range(hq):
        g = h // group
        for w in range(W):
            last = P + w
            logits = []
            for j in range(last + 1):
                dot = math.fsum(q_win[h][w][i] * K[g][j][i] for i in range(d))
                logits.append(dot / math.sqrt(d))
            top = max(logits)
            ex = [math.exp(x - top) for x in logits]
            tot = math.fsum(ex)
            for j in range(P):
                S[g][j] += ex[j] / tot
    return S


def pool(row, pool_k):
    half = pool_k // 2
    out = []
    for j in range(len(row)):
        neigh = [row[t] for t in range(j - half, j + half + 1) if 0 <= t < len(row)]
        out.append(max(neigh))
    return out


def select(pooled, k, n):
    P = len(pooled)
    ranked = sorted(range(P), key=lambda j: (-pooled[j], j))
    return sorted(ranked[:k]) + list(range(P, n))


def attention(q, Kc, Vc, length):
    """q[i]; Kc[j][i]; Vc[j][i] -> out[i] over the first ``length`` rows."""
    d = len(q)
    logits = [math.fsum(q[i] * Kc[j][i] for i in range(d)) / math.sqrt(d)
              for j in range(length)]
    top = max(logits)
    ex = [math.exp(x - top) for x in logits]
    tot = math.fsum(ex)
    return [math.fsum(ex[j] * Vc[j][i] for j in range(length)) / tot for i in range(d)]
