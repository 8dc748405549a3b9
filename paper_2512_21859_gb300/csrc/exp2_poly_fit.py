"""Derives the polynomial behind exp2_poly2 (csrc/tc_ptx.cuh).

2^f on [-0.5, 0.5] by a degree-5 polynomial minimising the largest relative
error (Remez exchange started from Chebyshev nodes), then rounded to fp32 and
checked under fp32 Horner evaluation. Run: python exp2_poly_fit.py
Printed: max relative error 7.5e-8 (exact arithmetic), 2.1e-7 (fp32 Horner).
"""
import numpy as np
# fit 2^f on [-0.5, 0.5] with a degree-5 polynomial minimising the max relative error:
# start from interpolation at Chebyshev nodes, then a few Remez exchange steps on the
# weighted error e(f) = (p(f) - 2^f) / 2^f.
deg = 5
a, b = -0.5, 0.5
def target(f): return np.exp2(f)
nodes = (a + b) / 2 + (b - a) / 2 * np.cos(np.pi * (2 * np.arange(deg + 2) + 1) / (2 * (deg + 2)))
nodes = np.sort(nodes)
grid = np.linspace(a, b, 200001)
for it in range(12):
    # solve p(x_i) - t(x_i) = (-1)^i E t(x_i)
    A = np.zeros((deg + 2, deg + 2))
    for i, x in enumerate(nodes):
        A[i, :deg + 1] = x ** np.arange(deg + 1)
        A[i, deg + 1] = -((-1) ** i) * target(x)
    sol = np.linalg.solve(A, target(nodes))
    c = sol[:deg + 1]
    err = (np.polyval(c[::-1], grid) - target(grid)) / target(grid)
    # new extrema: local maxima of |err| with alternating signs
    idx = [0] + [i for i in range(1, len(grid) - 1) if (abs(err[i]) >= abs(err[i-1]) and abs(err[i]) >= abs(err[i+1]))] + [len(grid) - 1]
    cand = sorted(idx, key=lambda i: grid[i])
    # pick deg+2 alternating extrema
    pts = []
    for i in cand:
        if pts and np.sign(err[i]) == np.sign(err[pts[-1]]):
            if abs(err[i]) > abs(err[pts[-1]]): pts[-1] = i
        else:
            pts.append(i)
    while len(pts) > deg + 2:
        if abs(err[pts[0]]) < abs(err[pts[-1]]): pts.pop(0)
        else: pts.pop()
    if len(pts) == deg + 2:
        nodes = grid[pts]
print("max rel err (fp64 poly):", np.max(np.abs(err)))
c32 = c.astype(np.float32)
print("coefficients c0..c5 (fp32):")
for v in c32: print("  %.9e  (0x%08x)" % (v, np.float32(v).view(np.uint32)))
# simulate fp32 evaluation with per-operation rounding (Horner, fused multiply-add emulated in fp64 then rounded)
def horner32(f):
    p = np.float32(c32[5])
    for k in range(4, -1, -1):
        p = np.float32(np.float64(p) * np.float64(f) + np.float64(c32[k]))
    return p
fs = np.linspace(-0.5, 0.5, 100001).astype(np.float32)
vals = np.array([horner32(f) for f in fs[::10]])
ref = np.exp2(fs[::10].astype(np.float64))
print("max rel err (fp32 Horner):", np.max(np.abs(vals.astype(np.float64) - ref) / ref))
