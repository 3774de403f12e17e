"""Pins of the oracle's Eq. 3 fit and Sec. 3.2 quantiser: the closed-form
weighted ridge solution from numpy's solver, the orthonormal special case
(ordinary least squares is a projection), exact scaling laws, the exponent rule
by brute force, and round-half-even codes from numpy."""
import numpy as np
import pytest


def _tile(rng, C, scale_r=1e-3, sigma_d=1.0):
    r = rng.normal(0, scale_r, C).astype(np.float32)
    d = rng.lognormal(0, sigma_d, C).astype(np.float32)
    return r, d


def _closed_form(C, P, ridge_rel, r, d, neg):
    B = np.where(neg.T == 1, -1.0, 1.0) / np.sqrt(C)
    r = r.astype(np.float64)
    d = d.astype(np.float64)
    eps = ridge_rel * d.mean()
    A = B.T @ (d[:, None] * B) + eps * np.eye(P)
    return np.linalg.solve(A, B.T @ (d * r)), np.linalg.cond(A)


@pytest.mark.parametrize("C,P", [(8, 2), (16, 4), (64, 4), (128, 2), (64, 8)])
def test_fit_matches_closed_form(orc, C, P):
    rng = np.random.default_rng(C * 10 + P)
    prm = orc.params(C=C, P=P, b=4, S=1, ridge_rel=1e-3)
    checked = 0
    for trial in range(60):
        r, d = _tile(rng, C)
        neg = orc.gen_basis(0, trial, C, P, 1)[3]
        ref, cond = _closed_form(C, P, 1e-3, r, d, neg)
        df = orc.def_fit(C, P, 1e-3, r, d, neg)
        assert np.allclose(df, ref, rtol=1e-10, atol=1e-16)
        out = orc.score_candidate(prm, r, d, neg)
        assert out is not None
        if cond < 1e3:
            scale = np.abs(ref).max()
            assert np.abs(out["alpha"] - ref).max() <= 2e-5 * scale
            checked += 1
    assert checked > 30


def test_uniform_weights_zero_ridge_is_orthogonal_projection(orc):
    """d = 1, eps = 0: G = I exactly, so alpha* = B^T r (ordinary LS on orthonormal columns)."""
    rng = np.random.default_rng(1)
    for C, P in [(16, 4), (64, 4), (128, 2)]:
        prm = orc.params(C=C, P=P, ridge_rel=0.0)
        for s in range(20):
            r = rng.normal(0, 1e-2, C).astype(np.float32)
            neg = orc.gen_basis(0, s, C, P, 1)[3]
            B = np.where(neg.T == 1, -1.0, 1.0) / np.sqrt(C)
            out = orc.score_candidate(prm, r, np.ones(C, np.float32), neg)
            proj = B.T @ r.astype(np.float64)
            assert np.allclose(out["alpha"], proj, rtol=0, atol=1e-6 * np.abs(r).sum())


def test_scaling_laws_are_exact(orc):
    """Scaling d by 2^k leaves fit and codes unchanged and scales the gain by 2^k;
    scaling r by 2^k shifts the exponent by k and scales the gain by 4^k."""
    rng = np.random.default_rng(2)
    prm = orc.params(C=64, P=4, b=4, ridge_rel=1e-4)
    for s in range(30):
        r, d = _tile(rng, 64)
        neg = orc.gen_basis(0, s, 64, 4, 1)[3]
        base = orc.score_candidate(prm, r, d, neg)
        dd = orc.score_candidate(prm, r, d * np.float32(8.0), neg)
        assert np.array_equal(dd["codes"], base["codes"]) and dd["scale"] == base["scale"]
        assert dd["gain"] == base["gain"] * 8.0
        rr = orc.score_candidate(prm, r * np.float32(0.25), d, neg)
        assert np.array_equal(rr["codes"], base["codes"]) and rr["scale"] == base["scale"] - 2
        assert rr["gain"] == base["gain"] / 16.0


def test_exponent_and_codes_pow2(orc):
    rng = np.random.default_rng(4)
    for b in (2, 3, 4, 6, 8):
        qmax = 2 ** (b - 1) - 1
        prm = orc.params(C=32, P=3, b=b, ridge_rel=1e-4)
        for s in range(40):
            r, d = _tile(rng, 32, scale_r=10 ** rng.uniform(-5, 0))
            neg = orc.gen_basis(0, s, 32, 3, 1)[3]
            out = orc.score_candidate(prm, r, d, neg)
            a = out["alpha"].astype(np.float64)
            amax = np.abs(a).max()
            e = out["scale"]
            # smallest integer e with amax <= qmax * 2^e (brute force over integers)
            smallest = next(k for k in range(-200, 200) if amax <= qmax * 2.0 ** k)
            assert e == smallest
            expect = np.clip(np.rint(a * 2.0 ** -e), -qmax, qmax)  # numpy rint: half to even
            assert np.array_equal(out["codes"], expect.astype(np.int64))


def test_exponent_field_clips_and_codes_stay_symmetric(orc):
    """A 2-bit exponent field holds e in [-2, 1]: an exponent outside it is
    clamped to the field and the codes to [-qmax, qmax], so a coefficient
    beyond the range gets +-qmax with its own sign, never -qmax - 1."""
    rng = np.random.default_rng(9)
    qmax = 7
    prm = orc.params(C=32, P=3, b=4, b_e=2, ridge_rel=1e-4)
    clipped_neg = clipped_low = 0
    for s in range(60):
        r, d = _tile(rng, 32, scale_r=10 ** rng.uniform(-4, 2))
        neg = orc.gen_basis(0, s, 32, 3, 1)[3]
        out = orc.score_candidate(prm, r, d, neg)
        a = out["alpha"].astype(np.float64)
        smallest = next(k for k in range(-200, 200) if np.abs(a).max() <= qmax * 2.0 ** k)
        e = min(max(smallest, -2), 1)
        assert out["scale"] == e
        x = a * 2.0 ** -e
        assert np.array_equal(out["codes"], np.clip(np.rint(x), -qmax, qmax).astype(np.int64))
        assert np.abs(out["codes"]).max() <= qmax
        clipped_neg += int((x < -qmax - 0.5).sum())
        clipped_low += int(smallest < -2)
    assert clipped_neg > 0 and clipped_low > 0     # both ends of the field were exercised


def test_codes_fp16_scale(orc):
    rng = np.random.default_rng(5)
    prm = orc.params(C=64, P=4, b=4, scale_mode=1, b_e=16, ridge_rel=1e-4)
    for s in range(40):
        r, d = _tile(rng, 64)
        neg = orc.gen_basis(0, s, 64, 4, 1)[3]
        out = orc.score_candidate(prm, r, d, neg)
        a = out["alpha"]
        sc = np.float16(np.float32(np.abs(a).max()) / np.float32(7.0))
        assert (out["scale"] & 0xFFFF) == int(np.array(sc).view(np.uint16))
        q = np.clip(np.rint(a / np.float32(sc)), -7, 7)
        assert np.array_equal(out["codes"], q.astype(np.int64))


def test_rtn_is_optimal_code_when_basis_orthonormal_under_weights(orc):
    """d = 1, eps = 0: the weighted error separates per coefficient, so for the
    chosen exponent the round-to-nearest codes beat every other code vector."""
    import itertools
    rng = np.random.default_rng(6)
    C, P, b = 8, 2, 3
    qmax = 3
    prm = orc.params(C=C, P=P, b=b, ridge_rel=0.0)
    ones = np.ones(C)
    for s in range(25):
        r = rng.normal(0, 1e-2, C).astype(np.float32)
        neg = orc.gen_basis(0, s, C, P, 1)[3]
        out = orc.score_candidate(prm, r, np.ones(C, np.float32), neg)
        sc = orc.scale_value(prm, out["scale"])
        g_rtn = orc.def_gain(C, P, r, ones, neg, out["codes"], sc)
        best = max(orc.def_gain(C, P, r, ones, neg, np.array(cv), sc)
                   for cv in itertools.product(range(-qmax, qmax + 1), repeat=P))
        assert g_rtn >= best - 1e-12 * abs(best)


def test_quantised_gain_never_exceeds_ls_optimum(orc):
    rng = np.random.default_rng(7)
    C, P = 16, 4
    prm = orc.params(C=C, P=P, b=4, ridge_rel=1e-6)
    for s in range(60):
        r, d = _tile(rng, C)
        neg = orc.gen_basis(0, s, C, P, 1)[3]
        out = orc.score_candidate(prm, r, d, neg)
        B = np.where(neg.T == 1, -1.0, 1.0) / np.sqrt(C)
        bv = B.T @ (d.astype(np.float64) * r)
        G = B.T @ (d.astype(np.float64)[:, None] * B)
        g_ls = bv @ np.linalg.solve(G, bv)
        g_q = orc.def_gain(C, P, r, d, neg, out["codes"], orc.scale_value(prm, out["scale"]))
        assert g_q <= g_ls * (1 + 1e-9)


def test_fixed_point_grid(orc):
    """q = ilogb(max|x|) - 20 and X = rint(x 2^-q) (numpy: frexp/ldexp/rint, half to even)."""
    rng = np.random.default_rng(8)
    for trial in range(200):
        scale = 10.0 ** rng.uniform(-30, 10)
        x = (rng.normal(0, 1, 64) * scale).astype(np.float32)
        if trial % 7 == 0:
            x[rng.integers(64)] = 0.0
        q, X = orc.fixed_point(x)
        m = np.abs(x).max()
        e = np.frexp(np.float64(m))[1] - 1          # ilogb
        assert q == e - 20
        want = np.rint(np.ldexp(x.astype(np.float64), -q))
        assert np.array_equal(X, want.astype(np.int32))
        assert np.abs(X).max() <= 2 ** 21 and np.abs(X).max() >= 2 ** 20
    assert orc.fixed_point(np.zeros(16, np.float32))[0] == 0
    q, X = orc.fixed_point(np.full(16, 1e-35, np.float32))      # below 2^-100: all zero
    assert q == 0 and not X.any()


def test_correlation_is_the_rounded_exact_sum(orc):
    """u_p = 2^q * RN(sum_j m_p(j) Y_j): recomputed here with exact Python integers,
    and within (C/2 + 1) 2^q of the real correlation sum_j m_p(j) y_j."""
    rng = np.random.default_rng(9)
    C, P = 64, 4
    prm = orc.params(C=C, P=P, ridge_rel=0.0)
    for s in range(30):
        r = rng.normal(0, 1e-3, C).astype(np.float32)
        neg = orc.gen_basis(0, s, C, P, 1)[3]
        out = orc.score_candidate(prm, r, np.ones(C, np.float32), neg)  # d = 1: G = I, alpha = b
        q, Y = orc.fixed_point(r)
        for p in range(P):
            exact = sum(int(-Y[j]) if neg[p, j] else int(Y[j]) for j in range(C))
            u = np.float32(np.ldexp(np.float32(exact), q))             # float32() rounds once
            assert out["alpha"][p] == np.float32(np.float32(1 / 8) * u)
            real = float(np.sum(np.where(neg[p] == 1, -1.0, 1.0) * r.astype(np.float64)))
            assert abs(float(u) - real) <= (C / 2 + 1) * 2.0 ** q
