"""Pins of the oracle's allocation (Sec. 3.3) and stream (Sec. 3.4) by their
invariants: positivity, rank order, quota and budget feasibility and
maximality, nested progressive prefixes, and a header/records round trip."""
import struct

import numpy as np
import pytest


def _cands(orc, rng, prm, shapes):
    out = []
    for rows, cols in shapes:
        W0 = rng.normal(0, 0.02, (rows, cols)).astype(np.float32)
        W = (W0 + rng.normal(0, 1e-3, (rows, cols))).astype(np.float32)
        act = rng.lognormal(0, 1.5, cols).astype(np.float32)
        F = rng.lognormal(0, 1.5, (rows, cols)).astype(np.float32)
        out.append(orc.encode_tiles(prm, W, W0, act, fisher=F, w_act=0.5, w_fisher=0.5))
    c = np.concatenate(out)
    # a few non-positive / invalid gains to exercise eligibility
    kill = rng.choice(len(c), len(c) // 20, replace=False)
    c["gain"][kill[: len(kill) // 2]] = -np.inf
    c["gain"][kill[len(kill) // 2:]] = -np.abs(c["gain"][kill[len(kill) // 2:]])
    return c


def _parse(orc, prm, stream, shapes):
    n_mod = len(shapes)
    h = orc.header_bytes(n_mod)
    magic, ver, var, smode, C, P, b, b_e, e_bias, perm, _, S, nm, gseed, K = struct.unpack_from(
        "<IHBBHBBBbBBIIQQ", stream, 0)
    assert (magic, ver, var, smode, C, P, b, b_e, e_bias, perm, S, nm, gseed) == (
        0x52535741, 1, prm.variant, prm.scale_mode, prm.C, prm.P, prm.b, prm.b_e, prm.e_bias,
        prm.permute, prm.S, n_mod, prm.gen_seed)
    mods = [struct.unpack_from("<II", stream, 40 + 8 * m) for m in range(n_mod)]
    T = sum(r * c // prm.C for r, c in shapes)
    L = orc.record_bytes(prm, T)
    assert len(stream) == h + K * L
    recs = [orc.unpack_record(prm, T, stream[h + k * L: h + (k + 1) * L]) for k in range(K)]
    return K, mods, recs


def test_u_per_module_quotas(orc):
    rng = np.random.default_rng(21)
    prm = orc.params(C=16, P=2, b=4, S=8, variant=0)
    shapes = [(32, 64), (8, 32), (64, 48)]
    cands = _cands(orc, rng, prm, shapes)
    rate = 0.9
    stream, counts, nbytes = orc.select_records(prm, shapes, cands, [rate])
    K, mods, recs = _parse(orc, prm, stream, shapes)
    N = sum(r * c for r, c in shapes)
    h = orc.header_bytes(len(shapes))
    T_m = [r * c // 16 for r, c in shapes]
    L = orc.record_bytes(prm, sum(T_m))
    B = orc.budget_bytes(rate, N)
    assert nbytes[0] == len(stream) <= B
    assert [m[0] for m in mods] == T_m and [m[1] for m in mods] == list(counts)
    off = np.cumsum([0] + T_m)
    k = 0
    for m, (rows, cols) in enumerate(shapes):
        mine = recs[k:k + counts[m]]
        k += counts[m]
        tiles = [t for t, _ in mine]
        assert all(off[m] <= t < off[m + 1] for t in tiles)
        gains = [float(cands[t]["gain"]) for t in tiles]
        assert all(g > 0 for g in gains)
        assert all(gains[i] > gains[i + 1] or (gains[i] == gains[i + 1] and tiles[i] < tiles[i + 1])
                   for i in range(len(tiles) - 1))
        pos = [t for t in range(off[m], off[m + 1]) if cands[t]["gain"] > 0]
        dropped = sorted(set(pos) - set(tiles))
        if dropped:
            assert max(cands["gain"][dropped]) <= min(gains) if gains else True
        # quota feasibility and maximality: proportional share of the byte budget
        share = (B - h) * rows * cols / N
        assert counts[m] * L <= share + 1e-9
        assert counts[m] == len(pos) or (counts[m] + 1) * L > share
        for t, c in mine:
            assert c["seed"] == cands[t]["seed"] and c["scale"] == cands[t]["scale"]
            assert np.array_equal(c["code"], cands[t]["code"])


def test_pf_progressive_prefixes_nest(orc):
    rng = np.random.default_rng(22)
    prm = orc.params(C=16, P=4, b=4, S=8, variant=1)
    shapes = [(16, 64), (32, 32)]
    cands = _cands(orc, rng, prm, shapes)
    rates = [0.5, 1.0, 2.0, 4.0]
    stream, counts, nbytes = orc.select_records(prm, shapes, cands, rates)
    K, mods, recs = _parse(orc, prm, stream, shapes)
    N = sum(r * c for r, c in shapes)
    T = sum(r * c // 16 for r, c in shapes)
    L = orc.record_bytes(prm, T)
    h = orc.header_bytes(2)
    npos = int((cands["gain"] > 0).sum())
    assert K == max(counts) and list(counts) == sorted(counts)
    for r, k, nb in zip(rates, counts, nbytes):
        B = orc.budget_bytes(r, N)
        assert nb == h + k * L <= B
        assert k == npos or nb + L > B
        # the single-rate stream is the same ranked prefix
        s1, c1, _ = orc.select_records(prm, shapes, cands, [r])
        assert c1[0] == k and s1[h:] == stream[h:h + k * L]
    gains = np.array([cands[t]["gain"] for t, _ in recs], np.float64)
    assert np.all(gains > 0) and np.all(np.diff(gains) <= 0)
    assert len({t for t, _ in recs}) == len(recs)
    # tiles disjoint: cumulative gain over nested prefixes is non-decreasing
    assert np.all(np.diff(np.cumsum(gains)) >= 0)
    # every eligible tile not in the stream ranks below the last one kept
    kept = {t for t, _ in recs}
    rest = [cands[t]["gain"] for t in range(T) if cands[t]["gain"] > 0 and t not in kept]
    if rest and recs:
        assert max(rest) <= gains[-1]
    assert sum(m[1] for m in mods) == K


def test_stream_never_exceeds_the_rate_budget(orc):
    """Eq. 5: the whole stream, header included, fits rate * N / 8 bytes. At
    211/512 bit/weight on 2048 weights the budget is 105.5 bytes: after the
    56-byte header nine 5-byte records (101 bytes) fit and a tenth (106) does
    not, for the progressive prefixes and for one module's quota alike."""
    rng = np.random.default_rng(23)
    shapes = [(16, 64), (32, 32)]
    rate = 211 / 512
    for variant in (1, 0):
        prm = orc.params(C=16, P=4, b=4, S=8, variant=variant)
        sh = shapes if variant == 1 else [(32, 64)]      # U: one module takes the whole budget
        cands = _cands(orc, rng, prm, sh)
        assert (cands["gain"] > 0).sum() >= 10
        assert orc.record_bytes(prm, 128) == 5 and orc.header_bytes(len(sh)) == 40 + 8 * len(sh)
        stream, counts, nbytes = orc.select_records(prm, sh, cands, [rate])
        h = 40 + 8 * len(sh)
        k = (105 - h) // 5                                # records that fit in 105.5 bytes
        assert int(counts.sum()) == k and int(nbytes[0]) == h + 5 * k <= 105.5 < h + 5 * (k + 1)
    # U over two equal modules at 105/256 bit/weight: B - h = 49 bytes, so each
    # module's quota is 24 bytes (4 records) and the stream 96 of 105 bytes
    prm = orc.params(C=16, P=4, b=4, S=8, variant=0)
    cands = _cands(orc, rng, prm, shapes)
    stream, counts, nbytes = orc.select_records(prm, shapes, cands, [105 / 256])
    assert list(counts) == [4, 4] and int(nbytes[0]) == 96


def test_zero_gains_never_make_records(orc):
    """Sec. 3.3: only a positive weighted error reduction earns a record, so
    candidates with a gain of exactly +0 or -0 are dropped even when the
    budget (16 bits/weight here) would hold every tile."""
    rng = np.random.default_rng(24)
    shapes = [(16, 64), (32, 32)]
    for variant in (0, 1):
        prm = orc.params(C=16, P=4, b=4, S=8, variant=variant)
        cands = _cands(orc, rng, prm, shapes)
        cands["gain"][::4] = 0.0
        cands["gain"][1::9] = -0.0
        npos = int((cands["gain"] > 0).sum())
        stream, counts, nbytes = orc.select_records(prm, shapes, cands, [16.0])
        K, mods, recs = _parse(orc, prm, stream, shapes)
        assert K == npos == int(counts.sum())
        assert all(cands[t]["gain"] > 0 for t, _ in recs)


def test_budget_below_header_is_an_error(orc):
    prm = orc.params(C=16, P=2, b=4, S=4)
    cands = np.zeros(4, orc.CANDIDATE_DTYPE)
    with pytest.raises(ValueError):
        orc.select_records(prm, [(4, 16)], cands, [1.0])   # 64 weights -> 8 B < 48 B header


def test_no_positive_gain_gives_empty_stream(orc):
    prm = orc.params(C=16, P=2, b=4, S=4)
    cands = np.zeros(64, orc.CANDIDATE_DTYPE)
    cands["gain"] = -np.inf
    stream, counts, nbytes = orc.select_records(prm, [(64, 16)], cands, [8.0])
    assert counts[0] == 0 and len(stream) == orc.header_bytes(1)


@pytest.mark.parametrize("variant", [0, 1])
def test_equal_gains_are_ranked_by_tile_ascending(orc, variant):
    """Ties in rho = gain / L (one L for every record) are broken by the global
    tile index, smallest first, in both allocations: with every gain drawn
    from three values and a budget that keeps part of each tie class, the
    stream lists each class's tiles in ascending order and keeps the smallest
    ones of the class that is cut."""
    prm = orc.params(C=16, P=2, b=4, S=4, variant=variant)
    shapes = [(64, 64)]
    T = 64 * 64 // 16
    rng = np.random.default_rng(31)
    cands = np.zeros(T, orc.CANDIDATE_DTYPE)
    cands["gain"] = rng.choice(np.array([1.0, 2.0, 3.0], np.float32), T)
    cands["seed"] = rng.integers(0, 4, T)
    stream, counts, _ = orc.select_records(prm, shapes, cands, [0.75])
    K, _, recs = _parse(orc, prm, stream, shapes)
    assert 0 < K < T
    tiles = [t for t, _ in recs]
    gains = [float(cands[t]["gain"]) for t in tiles]
    assert gains == sorted(gains, reverse=True)
    for g in set(gains):
        cls = [t for t, gg in zip(tiles, gains) if gg == g]
        assert cls == sorted(cls)
        everyone = np.flatnonzero(cands["gain"] == g)
        assert cls == sorted(everyone.tolist())[: len(cls)]   # the smallest tiles of the class
