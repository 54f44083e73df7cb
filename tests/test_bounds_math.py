"""The row bounds behind the last hop's skip and the two-hop reach path,
checked in exact (fp64) arithmetic against the oracle's propagated scores.

With u >= 0 and w >= 0, s^(H) = u * sum_{h=0..H} (alpha R)^h (the hop
recursion s^(h) = u + alpha s^(h-1) R of §4.1), and the mass levels
M^(0) = 1, M^(t) = M^(t-1) R (in-weight sums of the previous level):

  L0_j + Lmin sum_{t=1..H} alpha^t M^(t)_j  <=  s^(H)_{j,b}
                                              <=  U0_j + Umax sum_t alpha^t M^(t)_j

for every row j and query b, where U0 / L0 are the row's largest / smallest
u over the queries and Umax / Lmin their extremes over the rows that have
out-edges (the only sources).  The device evaluates the same sums in fp32
and widens them by the rounding bound of each sum; here the inequalities are
checked without that margin.  A dropped term, a transposed R (out- instead
of in-weights) or a wrong extreme makes one of them fail.
"""
import math

import numpy as np
import pytest

import oracle
from test_oracle_pins import dense_R, softmax_lib, tiny_store, widen


def _case(seed, n, deg, alpha, hops, empty_rows):
    emb, q, row_ptr, col, aff = tiny_store(seed, n, 16, deg, n_q=9, empty_rows=empty_rows)
    w = oracle.row_softmax(row_ptr, aff)
    out = oracle.retrieve(emb, q, row_ptr, col, w, tau=0.5, alpha=alpha, hops=hops, k=8,
                          want_final=True)
    R = dense_R(n, row_ptr, col, w)
    # the normalised first-level scores u/Z (the bounds are per-query scale free)
    z = 0.5 * widen(q) @ widen(emb).T
    u = np.stack([softmax_lib(z[b]) for b in range(z.shape[0])])
    return out, R, u, row_ptr


@pytest.mark.parametrize("hops,alpha", [(1, 0.5), (2, 0.5), (3, 0.4), (2, 1.0), (16, 0.6)])
@pytest.mark.parametrize("empty_rows", [False, True])
def test_row_bounds_bracket_propagated_scores(hops, alpha, empty_rows):
    out, R, u, row_ptr = _case(11, 90, 6, alpha, hops, empty_rows)
    n = R.shape[0]
    s = out["final"]                                   # [B][n], s^(H) / Z
    u0, l0 = u.max(axis=0), u.min(axis=0)
    sources = np.diff(row_ptr) > 0
    umax, lmin = u0.max(), l0[sources].min()
    M = [np.ones(n)]
    for _ in range(hops):
        M.append(M[-1] @ R)
    c = sum(alpha ** t * M[t] for t in range(1, hops + 1))
    ub, lb = u0 + umax * c, l0 + lmin * c
    tol = 1e-12
    assert (s <= ub[None, :] * (1 + tol)).all()
    assert (s >= lb[None, :] * (1 - tol)).all()


@pytest.mark.parametrize("hops", [1, 2])
def test_floor_is_below_every_kth_score(hops):
    """The skip's floor, the k-th largest lower bound over any subset of the
    rows, never exceeds a query's k-th largest final score; every row whose
    upper bound is below it is outside every query's top-k."""
    alpha, k = 0.5, 8
    out, R, u, row_ptr = _case(12, 120, 7, alpha, hops, False)
    n = R.shape[0]
    s = out["final"]
    u0, l0 = u.max(axis=0), u.min(axis=0)
    umax, lmin = u0.max(), l0.min()
    M = [np.ones(n)]
    for _ in range(hops):
        M.append(M[-1] @ R)
    c = sum(alpha ** t * M[t] for t in range(1, hops + 1))
    ub, lb = u0 + umax * c, l0 + lmin * c
    heavy = np.argsort(-np.array(M[1]))[:40]           # a subset: the heaviest rows
    floor = np.sort(lb[heavy])[::-1][k - 1]
    kth = np.sort(s, axis=1)[:, ::-1][:, k - 1]
    assert (floor <= kth * (1 + 1e-12)).all()
    pruned = np.nonzero(ub < floor)[0]
    for b in range(s.shape[0]):
        assert not set(pruned.tolist()) & set(out["ids"][b].tolist())


@pytest.mark.parametrize("hops,alpha", [(1, 0.5), (2, 0.5), (2, 1.0), (3, 0.4)])
def test_reach_coefficients_reproduce_propagated_scores(hops, alpha):
    """The unrolled recursion behind the two-hop path.  With the graph-only
    reach coefficients C_1[k][j] = w(k -> j) (column j: row j's in-weights)
    and C_t = R C_{t-1} (row k: k's out-edges applied to the previous
    level), s^(H)_j = u_j + sum_t alpha^t sum_k C_t[k][j] u_k for every row
    and query: the oracle's propagated scores.  Only the candidates' columns
    are ever needed, and each column follows the recursion on its own.  A
    transposed C_1 (out- instead of in-weights) fails."""
    out, R, u, _ = _case(13, 80, 5, alpha, hops, True)
    s = out["final"]
    C = [R.copy()]
    for _ in range(2, hops + 1):
        C.append(R @ C[-1])
    got = u + sum(alpha ** (t + 1) * (u @ C[t]) for t in range(hops))
    np.testing.assert_allclose(got, s, rtol=1e-12, atol=0)
    # the same for a subset of columns, computed column by column
    cols = [3, 17, 41]
    Csub = [R[:, cols]]
    for _ in range(2, hops + 1):
        Csub.append(R @ Csub[-1])
    sub = u[:, cols] + sum(alpha ** (t + 1) * (u @ Csub[t]) for t in range(hops))
    np.testing.assert_allclose(sub, s[:, cols], rtol=1e-12, atol=0)
    # planted: out-weights in place of in-weights
    bad = u + sum(alpha ** (t + 1) * (u @ np.linalg.matrix_power(R.T, t + 1)) for t in range(hops))
    assert not np.allclose(bad, s, rtol=1e-6, atol=0)


# --------------------------------------------------------------------------- fp32 margins
F32 = np.float32


def _x(n):
    """The per-level rounding allowance of a row with n in-edges, as the
    device computes it in fp32: 3.25 (n + 8) 2^-24."""
    return F32(3.25) * F32(n + 8) * F32(5.9604645e-8)


def _seq_sum_f32(w, a):
    """A worse evaluation than the device's: every product rounded to fp32,
    then one sequential fp32 chain over all n terms (the device fuses each
    product into its sum and splits the chain over lanes and segments)."""
    return np.cumsum((w * a).astype(F32), dtype=F32)[-1]


@pytest.mark.parametrize("n", [1, 7, 256, 4096, 100_000, 818_357])
@pytest.mark.parametrize("kind", ["uniform", "lognormal", "constant"])
def test_level_margins_cover_fp32_sums(n, kind):
    """One mass level in fp32: the device's widened sums, Σ·(1 + x + x²)·(1 + 4e-6)
    above and Σ·(1 − x)·(1 − 4e-6) below, bracket the exact sum of the same fp32
    inputs, for in-degrees up to the largest hub of the 1M-chunk graph."""
    rng = np.random.default_rng(n)
    if kind == "uniform":
        w, a = rng.random(n).astype(F32), (1 + 10 * rng.random(n)).astype(F32)
    elif kind == "lognormal":
        w, a = rng.random(n).astype(F32), rng.lognormal(0, 2, n).astype(F32)
    else:
        w, a = np.full(n, 0.1, F32), np.full(n, 3.3, F32)
    exact = math.fsum((w.astype(np.float64) * a.astype(np.float64)).tolist())
    s = _seq_sum_f32(w, a)
    x = _x(n)
    up = F32(F32(s * F32(F32(1) + x + x * x)) * F32(1 + 4e-6))
    dn = F32(F32(s * F32(F32(1) - x)) * F32(1 - 4e-6))
    assert float(up) >= exact
    assert float(dn) <= exact


@pytest.mark.parametrize("hops", [1, 2, 16])
def test_final_bound_margin_covers_fp32_horner(hops):
    """The per-call bounds in fp32, ub = (U0 + Umax·Σ_t α^t M_t)(1 + 1e-5) by
    Horner's rule and lb likewise with (1 − 1e-5), bracket the exact value of
    the same fp32 inputs, up to sixteen hops."""
    rng = np.random.default_rng(hops)
    for _ in range(2000):
        alpha = F32(rng.random())
        M = rng.lognormal(2, 2, hops).astype(F32)
        u0, umax = F32(rng.random() * 1e-3), F32(rng.random())
        cu = F32(0)
        for t in range(hops, 0, -1):
            cu = F32(alpha * F32(cu + M[t - 1]))
        ub = F32(F32(umax * cu + u0) * F32(1 + 1e-5))      # fmaf: one rounding, a
        lb = F32(F32(umax * cu + u0) * F32(1 - 1e-5))      # second here is worse
        exact = float(u0) + float(umax) * sum(float(alpha) ** t * float(M[t - 1])
                                              for t in range(1, hops + 1))
        assert float(ub) >= exact and float(lb) <= exact


def test_fp32_hops_never_lower_a_score():
    """The fused filter's bound: with w >= 0 and alpha >= 0, s^(h) >= s^(h-1)
    elementwise also in fp32 when every hop sums a row's in-edges in the same
    order (each fma and add is monotone in its arguments), so the k-th
    largest sampled value of s^(H-1) is a safe threshold for s^(H).  Emulated
    with fp32 numpy, one sequential fma-free chain per row (product rounded,
    then added), for 12 hops."""
    out, R, u, row_ptr = _case(21, 150, 9, 0.9, 1, True)
    n = R.shape[0]
    u32 = u.astype(F32)
    alpha = F32(0.9)
    Rt = R.T.astype(F32)                                 # Rt[j][i] = w(i -> j)
    prev = u32.copy()
    for _ in range(12):
        nxt = np.empty_like(prev)
        for j in range(n):
            src = np.nonzero(Rt[j])[0]
            acc = np.zeros(prev.shape[0], F32)
            for i in src:                                 # the same order every hop
                acc = (acc + (Rt[j, i] * prev[:, i]).astype(F32)).astype(F32)
            nxt[:, j] = (u32[:, j] + (alpha * acc).astype(F32)).astype(F32)
        assert (nxt >= prev).all()
        prev = nxt


def _bf16_rne(x):
    """float32 -> nearest bf16 (ties to even), as float32 (bit arithmetic)."""
    b = np.ascontiguousarray(x, dtype=F32).view(np.uint32)
    r = (b + np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1))) & np.uint32(0xFFFF0000)
    return r.view(F32)


@pytest.mark.parametrize("seed", [0, 1])
def test_split_bf16_products_keep_the_candidates_terms(seed):
    """The candidates' two-hop terms sum_k coef[k][i] u[k][b] are computed on
    the tensor cores from split-bf16 operands: x = hi + lo with hi = bf16(x)
    and lo = bf16(x - hi) (x - hi is exact in fp32), and the three products
    hi*hi + hi*lo + lo*hi.  bf16 rounds to 8 significant bits, so
    |x - hi| <= 2^-8 |x| and |x - hi - lo| <= 2^-8 |x - hi| <= 2^-16 |x|; the
    dropped lo*lo is at most 2^-16 of the product; every product is thus
    within 3 * 2^-16 (4.6e-5) relative, and, all terms being non-negative,
    so is the sum: inside the 1e-4 near-tie band of the selection, where a
    single bf16 product (2^-8) is not.  The rounding errors have random
    signs, so the sums land far closer (below 1e-5 here).  Emulated with the
    products in fp64, on scores u = exp(tau <q, e> - c) of unit vectors
    (tau = 1/sqrt(d)) and heavy-tailed non-negative coefficients."""
    rng = np.random.default_rng(seed)
    n, d, nq, nk = 4096, 256, 16, 40
    e = rng.standard_normal((n, d)).astype(F32)
    e /= np.linalg.norm(e, axis=1, keepdims=True)
    q = rng.standard_normal((nq, d)).astype(F32)
    q /= np.linalg.norm(q, axis=1, keepdims=True)
    tau = 1.0 / math.sqrt(d)
    u = np.exp((tau * (e @ q.T) - tau).astype(F32)).astype(F32)          # [n][nq]
    coef = (rng.lognormal(-6.0, 2.0, (n, nk)) * (rng.random((n, nk)) < 0.3)).astype(F32)
    exact = coef.astype(np.float64).T @ u.astype(np.float64)            # [nk][nq]

    def split(x):
        hi = _bf16_rne(x)
        lo = _bf16_rne((x - hi).astype(F32))
        return hi.astype(np.float64), lo.astype(np.float64)

    ch, cl = split(coef)
    uh, ul = split(u)
    three = ch.T @ uh + ch.T @ ul + cl.T @ uh
    one = ch.T @ uh
    rel3 = np.abs(three - exact) / exact
    rel1 = np.abs(one - exact) / exact
    assert rel3.max() <= 3 * 2.0 ** -16, rel3.max()
    assert rel3.max() < 1e-5
    assert rel1.max() > 1e-4          # a single bf16 product would break the band
    # the split itself: hi + lo within 2^-16 of every operand
    assert (np.abs(ch + cl - coef) <= 2.0 ** -16 * coef).all()
    assert (np.abs(uh + ul - u) <= 2.0 ** -16 * u).all()
