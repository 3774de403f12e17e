"""Pin of the inequality behind the GPU search's exact pruning (Eq. 3, Eq. 4).

For any coefficients x the Eq. 4 gain 2 x^T b - x^T G x is at most
U_G = b^T G^-1 b, its maximum over x, and U_G <= (1 + eps tr(G^-1)) U_eps
with U_eps = b^T (G + eps I)^-1 b. The search skips a candidate when
U_eps m < g_best with m = (1 + eps tr(G^-1)) (1 + 2^-10 + 2^-14 kappa),
kappa = tr(G) tr(G^-1). Here b and G are rebuilt in numpy exactly as the
binary32 recipe stores them, U_eps is solved in double, and every quantised
gain the oracle reports must lie at or below U_eps m, including on tiles with
heavy-tailed, tiny and zero weights and with a large ridge."""
import numpy as np
import pytest

C, P = 64, 4


def stored_b_G(orc, r, d, neg, ridge_rel):
    """b and G (+ eps) as the recipe stores them: exact integer sums on the
    tile's fixed-point grids, rounded once, scaled by powers of two."""
    f32 = np.float32
    y = (d.astype(f32) * r.astype(f32)).astype(f32)
    qy, Y = orc.fixed_point(y)
    qd, D = orc.fixed_point(d.astype(f32))
    sgn = np.where(neg == 1, -1, 1).astype(np.int64)            # P x C
    c, c2 = f32(0.125), f32(1.0 / 64)
    S = (sgn * Y.astype(np.int64)).sum(1)
    b = (c * (np.array([np.ldexp(f32(s), qy) for s in S], f32))).astype(f32)
    two_qd = f32(np.ldexp(1.0, qd))
    gd = c2 * f32(f32(D.astype(np.int64).sum()) * two_qd)
    G = np.zeros((P, P))
    for p in range(P):
        G[p, p] = gd
        for q in range(p):
            v = (sgn[p] * sgn[q] * D.astype(np.int64)).sum()
            G[p, q] = G[q, p] = c2 * f32(f32(v) * two_qd)
    eps = float(f32(f32(ridge_rel) * gd))
    return b.astype(np.float64), G, eps


def multiplier(G, eps):
    try:
        np.linalg.cholesky(G)
        tri = np.trace(np.linalg.inv(G))
    except np.linalg.LinAlgError:
        return np.inf
    kappa = np.trace(G) * tri
    if not kappa <= 65536.0:
        return np.inf
    return (1 + eps * tri) * (1 + 2.0 ** -10 + 2.0 ** -14 * kappa)


def tiles(rng):
    """(r, d) pairs: Qwen-like residuals with t4 outliers and activation moments,
    heavy-tailed d, d with many exact zeros, and tiny/large magnitudes."""
    for k in range(24):
        r = (rng.normal(0, 2e-3, C) * (1 + 7 * (rng.random(C) < 0.02))).astype(np.float32)
        kind = k % 4
        if kind == 0:
            d = rng.lognormal(0, 1.0, C)
        elif kind == 1:
            d = 10.0 ** rng.uniform(-6, 6, C)                     # ill-conditioned G
        elif kind == 2:
            d = rng.lognormal(0, 1.0, C) * (rng.random(C) < 0.15)  # mostly zero weights
        else:
            d = rng.lognormal(0, 0.3, C)
            r = (r * 10.0 ** rng.uniform(-20, 3)).astype(np.float32)
        yield r, d.astype(np.float32)


@pytest.mark.parametrize("ridge_rel", [1e-6, 0.0, 0.5])
def test_quantised_gain_never_exceeds_the_pruning_bound(orc, ridge_rel):
    rng = np.random.default_rng(int(ridge_rel * 1e6) + 11)
    prm = orc.params(C=C, P=P, b=4, S=64, ridge_rel=ridge_rel)
    checked = finite_bounds = 0
    for r, d in tiles(rng):
        for s in range(64):
            neg = orc.gen_basis(0, s, C, P, 1)[3]
            out = orc.score_candidate(prm, r, d, neg)
            if out is None or not np.isfinite(out["gain"]):
                continue
            b, G, eps = stored_b_G(orc, r, d, neg, ridge_rel)
            m = multiplier(G, eps)
            checked += 1
            if not np.isfinite(m):
                continue
            finite_bounds += 1
            U = b @ np.linalg.solve(G + eps * np.eye(P), b)
            assert float(out["gain"]) <= U * m, (s, float(out["gain"]), U, m)
    assert checked > 1000 and finite_bounds > 0.5 * checked


def test_bound_is_tight_on_typical_tiles(orc):
    """The bound must also prune: on Qwen-like tiles U_eps m stays within 1% of
    the unquantised optimum U_G for most seeds (kappa is small)."""
    rng = np.random.default_rng(5)
    ratios = []
    for _ in range(8):
        r = rng.normal(0, 2e-3, C).astype(np.float32)
        d = rng.lognormal(0, 1.0, C).astype(np.float32)
        for s in range(32):
            neg = orc.gen_basis(0, s, C, P, 1)[3]
            b, G, eps = stored_b_G(orc, r, d, neg, 1e-6)
            m = multiplier(G, eps)
            U = b @ np.linalg.solve(G + eps * np.eye(P), b)
            ratios.append(U * m / (b @ np.linalg.solve(G, b)))
    assert np.median(ratios) < 1.01 and min(ratios) >= 1.0


def multiplier_binary32(gd, Goff, eps):
    """The multiplier as the GPU table builder evaluates it: LDL^T of G and the
    inverse trace in binary32 (fused multiply-adds emulated by one rounding of
    the double-precision result), the trace inflated by 1.5, the last steps
    rounded up (emulated by one step towards +inf after rounding)."""
    f = np.float32
    up = lambda x: np.nextafter(f(x), f(np.inf))
    fma = lambda a, b, c: f(np.float64(a) * np.float64(b) + np.float64(c))
    L = np.zeros((P, P), np.float32)
    d = np.zeros(P, np.float32)
    inv = np.zeros(P, np.float32)
    for k in range(P):
        dk = f(gd)
        for i in range(k):
            dk = fma(-f(L[k, i] * L[k, i]), d[i], dk)
        if not dk > 0:
            return np.inf
        d[k], inv[k] = dk, f(1.0 / np.float64(dk))
        for j in range(k + 1, P):
            v = f(Goff[j][k])
            for i in range(k):
                v = fma(-f(L[j, i] * L[k, i]), d[i], v)
            L[j, k] = f(v * inv[k])
    tr = f(0)
    for i in range(P):
        x = np.zeros(P, np.float32)
        x[i] = 1
        tr = f(tr + inv[i])
        for k in range(i + 1, P):
            v = f(0)
            for j in range(i, k):
                v = fma(-L[k, j], x[j], v)
            x[k] = v
            tr = fma(f(v * v), inv[k], tr)
    kappa = f(f(P * f(gd)) * tr)
    if not (tr > 0 and kappa <= 65536):
        return np.inf
    ts = up(1.5 * np.float64(tr))
    ks = up(1.5 * np.float64(up(np.float64(up(P * np.float64(gd))) * tr)))
    f1 = up(np.float64(eps) * ts + 1)
    f2 = up(2.0 ** -14 * np.float64(ks) + (1 + 2.0 ** -10))
    return float(up(np.float64(f1) * f2))


def test_binary32_multiplier_is_never_below_the_double_one():
    """The GPU builds the pruning multiplier in binary32 with a 1.5 safety factor
    on tr(G^-1); over Gram matrices of +-1 atoms under weights spanning twelve
    decades (condition numbers up to the 2^16 cutoff) it must stay at or above
    the double-precision multiplier, or be +inf (no pruning)."""
    rng = np.random.default_rng(17)
    checked, kappas = 0, []
    for trial in range(4000):
        scale = 10.0 ** rng.uniform(-6, 6)
        kind = trial % 4
        if kind == 0:
            dv = rng.lognormal(0, 2.0, C)
        elif kind == 1:
            dv = 10.0 ** rng.uniform(-6, 6, C)
        elif kind == 2:
            dv = rng.lognormal(0, 1.0, C) * (rng.random(C) < 0.2)
        else:  # weight on a few coordinates over a small floor: G nearly rank-deficient
            dv = np.full(C, 10.0 ** rng.uniform(-6, -2))
            dv[rng.choice(C, rng.integers(2, 5), replace=False)] = 1.0
        dv = (dv * scale).astype(np.float32).astype(np.float64)
        sgn = rng.choice([-1.0, 1.0], size=(P, C))
        G = (sgn * dv) @ sgn.T / C
        G = G.astype(np.float32).astype(np.float64)
        gd = float(np.float32(dv.sum() / C))
        np.fill_diagonal(G, gd)
        eps = float(np.float32(np.float32(1e-6) * np.float32(gd)))
        m64 = multiplier(G, eps)
        m32 = multiplier_binary32(gd, G, eps)
        if not np.isfinite(m32):
            continue
        checked += 1
        kappas.append(np.trace(G) * np.trace(np.linalg.inv(G)))
        assert np.isfinite(m64) and m32 >= m64, (trial, m32, m64)
    kappas = np.array(kappas)
    assert checked > 1000 and (kappas > 1e3).sum() >= 50 and (kappas > 1e4).sum() >= 10
