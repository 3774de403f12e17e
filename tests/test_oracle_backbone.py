"""Pins of the oracle's RTN-INT4 backbone (Eq. 1's W0 = Q(W), round to nearest
with groups of 128 inputs, Sec. 4), its scale double quantisation (SDQ,
Sec. 3.3) and the definition of the packed product (W0 + r_hat) x: an
independent torch implementation of RTN, the round-to-nearest error bound,
code ranges, exact sign and power-of-two scaling laws, the SDQ error bound and
its degenerate block, the metadata byte count, numpy's matmul, and the
oracle decoder."""
import numpy as np
import pytest
import torch


def _weights(rng, rows, cols, zero_groups=True):
    W = rng.normal(0, 0.02, (rows, cols)).astype(np.float32)
    W[:, rng.choice(cols, max(1, cols // 100), replace=False)] *= 8.0
    if zero_groups:
        W[0, :128] = 0.0                    # an all-zero group
        W[1, 128:256] = -0.0
    return W


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_rtn_matches_torch_restatement(orc, dtype):
    """Without SDQ the oracle's W0 equals the torch RTN used to build the
    benchmark's inputs (written separately), bit for bit."""
    from synth.workloads import rtn_int4_g128
    rng = np.random.default_rng(1)
    W = torch.from_numpy(_weights(rng, 40, 512)).to(dtype)
    got = orc.rtn_quantize(W.float().numpy())
    want = rtn_int4_g128(W).numpy()
    assert np.array_equal(got["W0"], want)  # as values: the torch product keeps a -0 that integer codes cannot


def test_rtn_error_bound_and_code_range(orc):
    rng = np.random.default_rng(2)
    W = _weights(rng, 64, 1024)
    r = orc.rtn_quantize(W)
    q, s = r["q"].reshape(-1, 128), r["s_eff"]
    w = W.reshape(-1, 128)
    assert q.min() >= -7 and q.max() <= 7              # |w/s| <= 7 (1 + 2^-11): never the -8 end
    nz = s > 0
    assert (np.abs(q[nz]).max(axis=1) == 7).all()     # the group's largest weight maps to +-7
    assert not q[~nz].any() and not r["W0"].reshape(-1, 128)[~nz].any()
    err = np.abs(w.astype(np.float64) - q * s[:, None].astype(np.float64))
    assert (err <= s[:, None] * 0.5 * (1 + 2.0 ** -20)).all()
    amax = np.abs(w).max(axis=1)
    assert np.array_equal(r["s16"], (amax / np.float32(7)).astype(np.float16).view(np.uint16))


def test_rtn_sign_and_power_of_two_laws(orc):
    rng = np.random.default_rng(3)
    W = _weights(rng, 16, 256, zero_groups=False)
    a, b = orc.rtn_quantize(W), orc.rtn_quantize(-W)
    assert np.array_equal(b["q"], -a["q"]) and np.array_equal(b["s16"], a["s16"])
    for sdq in (False, True):
        a = orc.rtn_quantize(W, sdq=sdq, block=8)
        c = orc.rtn_quantize(W * np.float32(4.0), sdq=sdq, block=8)
        assert np.array_equal(c["q"], a["q"])
        assert np.array_equal(c["s_eff"], a["s_eff"] * np.float32(4.0))
        assert np.array_equal(c["W0"], a["W0"] * np.float32(4.0))


def test_sdq_error_bound_and_constant_block(orc):
    rng = np.random.default_rng(4)
    W = _weights(rng, 64, 2048)
    plain, dq = orc.rtn_quantize(W), orc.rtn_quantize(W, sdq=True, block=256)
    s, st = plain["s_eff"].astype(np.float64), dq["s_eff"].astype(np.float64)
    G = len(s)
    mu, step = dq["consts"][0::2].astype(np.float64), dq["consts"][1::2].astype(np.float64)
    blk = np.arange(G) // 256
    assert np.abs(dq["c8"].astype(np.int64)).max() <= 127
    assert (np.abs(st - s) <= 0.5 * step[blk] + 4 * np.spacing(np.float32(s.max()))).all()
    for b in range(len(mu)):                         # mu is the block mean, rounded once
        m = s[blk == b].mean()
        assert abs(mu[b] - m) <= np.spacing(np.float32(m))
    # identical scales: the block is represented exactly
    Wc = np.tile(np.concatenate([np.full(127, 0.01, np.float32), [0.07]]), (8, 4)).astype(np.float32)
    r = orc.rtn_quantize(Wc, sdq=True, block=16)
    assert not r["c8"].any() and r["consts"][1] == 0.0
    assert np.array_equal(r["s_eff"], orc.rtn_quantize(Wc)["s_eff"])
    # the codes are still the first-level ones
    assert np.array_equal(dq["q"], plain["q"])


def test_rtn_divides_by_the_scale(orc):
    """The codes are rint(w / s_g) with the correctly rounded binary32 quotient
    (numpy's division), ties to even. With s_g = 7 * 2^-10 (a group whose
    largest weight is 7 s_g) the weights +-6.5 s_g are exact ties and give +-6,
    where a product with the rounded reciprocal 1/s_g would give +-7."""
    s = np.float32(0.0068359375)
    w = np.zeros((1, 128), np.float32)
    w[0, :4] = [7 * s, 0.04443359375, -0.04443359375, 0.02392577938735485]
    out = orc.rtn_quantize(w)
    assert out["s_eff"][0] == s
    expect = np.rint(w[0, :4] / s)
    assert list(expect) == [7, 6, -6, 3]
    assert list(out["q"].reshape(-1)[:4]) == list(expect)


def test_sdq_extreme_deviation_below_the_mean(orc):
    """One block where the scale farthest from the mean lies below it (a group
    of tiny weights among ordinary ones): its step still covers that deviation,
    so every reconstructed scale is within half a step of its own."""
    rng = np.random.default_rng(7)
    W = rng.normal(0, 0.02, (16, 2048)).astype(np.float32)    # 256 groups, one block
    W[5, 640:768] *= 1e-3
    plain, dq = orc.rtn_quantize(W), orc.rtn_quantize(W, sdq=True, block=256)
    s, st = plain["s_eff"].astype(np.float64), dq["s_eff"].astype(np.float64)
    mu, step = float(dq["consts"][0]), float(dq["consts"][1])
    assert np.argmax(np.abs(s - mu)) == 5 * 16 + 5 and s[5 * 16 + 5] < mu
    assert (np.abs(st - s) <= 0.5 * step + 4 * np.spacing(np.float32(s.max()))).all()


def test_sdq_short_last_block(orc):
    """A last block with fewer than 256 groups: its constant is the mean of its
    own n scales (numpy's mean, rounded once), and a short block of equal
    scales is reproduced exactly (their mean is that scale, the step is 0)."""
    rng = np.random.default_rng(6)
    W = _weights(rng, 64, 2176)                       # 17 groups a row: G = 1088 = 4 * 256 + 64
    plain, dq = orc.rtn_quantize(W), orc.rtn_quantize(W, sdq=True, block=256)
    s = plain["s_eff"].astype(np.float64)
    mu = dq["consts"][0::2].astype(np.float64)
    assert len(s) == 1088 and len(mu) == 5
    m = s[1024:].mean()
    assert abs(mu[4] - m) <= np.spacing(np.float32(m))
    # 3 groups a row, blocks of 16 over 8 rows: G = 24 = 16 + 8, every scale equal
    Wc = np.tile(np.concatenate([np.full(127, 0.01, np.float32), [0.07]]), (8, 3)).astype(np.float32)
    r = orc.rtn_quantize(Wc, sdq=True, block=16)
    assert len(r["consts"]) == 4 and not r["c8"].any() and r["consts"][3] == 0.0
    assert np.array_equal(r["s_eff"], orc.rtn_quantize(Wc)["s_eff"])


def test_backbone_metadata_bytes():
    """FP16 group scales cost 16 bits per 128 weights (0.125 bpw, Sec. 3.3);
    SDQ with 8-bit codes and a binary32 (mean, step) pair per 256 groups costs
    (8 + 64/256)/128 = 0.064453125 bpw on whole blocks (the paper reports
    0.068 without giving its format)."""
    rows, cols = 11008, 2048
    G = rows * cols // 128
    fp16 = 2 * G
    sdq = G + 8 * ((G + 255) // 256)
    assert fp16 * 8 / (rows * cols) == 0.125
    assert sdq == 176128 + 8 * 688 and abs(sdq * 8 / (rows * cols) - 0.064453125) < 1e-12


def test_packed_product_definition(orc):
    """K = 0: y = W0 x (numpy matmul of the oracle's W0). With records: within
    the rounding of the oracle decoder's binary32 W_hat of y (and of yabs)."""
    rng = np.random.default_rng(5)
    rows, cols = 48, 256
    W = _weights(rng, rows, cols, zero_groups=False)
    bb = orc.rtn_quantize(W, sdq=True, block=16)
    x = rng.normal(0, 1, (3, cols)).astype(np.float32)
    prm = orc.params(C=64, P=4, b=4, S=64)
    y0, a0, bad = orc.packed_gemv(prm, bb["q"], bb["s_eff"], 128, b"\0" * 48, 0, x)
    assert bad == 0
    ref = x.astype(np.float64) @ bb["W0"].astype(np.float64).T
    assert np.allclose(y0, ref, rtol=0, atol=1e-12 * a0.max())
    # a real stream: encode the residual W - W0 and select at 2 bits/weight
    d = (rng.lognormal(0, 1, cols) ** 2).astype(np.float32)
    cands = orc.encode_tiles(prm, W, bb["W0"], d)
    stream, counts, _ = orc.select_records(prm, [(rows, cols)], cands, [2.0])
    K = int(counts.sum())
    assert K > 0
    y, yabs, bad = orc.packed_gemv(prm, bb["q"], bb["s_eff"], 128, stream, K, x)
    assert bad == 0
    dec, _ = orc.decode_apply(prm, [bb["W0"]], stream, K)
    ref = x.astype(np.float64) @ dec[0].astype(np.float64).T
    assert (np.abs(y - ref) <= 2.0 ** -22 * yabs + 1e-30).all()
    assert (yabs >= np.abs(y)).all() and not np.allclose(y, y0)
    # yabs sums the backbone's and the residual's magnitudes separately; the
    # residual is the decoded weights less W0 (both binary32, so within one
    # rounding of the decoded weight)
    W0d = bb["W0"].astype(np.float64)
    R = dec[0].astype(np.float64) - W0d
    xa = np.abs(x.astype(np.float64))
    want = xa @ np.abs(W0d).T + xa @ np.abs(R).T
    assert (np.abs(yabs - want) <= 2.0 ** -22 * (xa @ np.abs(dec[0].astype(np.float64)).T) + 1e-30).all()
    assert (want - xa @ np.abs(W0d + R).T > 2.0 ** -18 * want).any()  # the two magnitudes differ here


def test_packed_product_repeated_tile_takes_later_record(orc):
    """A stream that names a tile twice (never written by the encoder): the
    product applies only the later record, as the decoder does, i.e. it equals
    the product of the stream without the earlier record."""
    rng = np.random.default_rng(7)
    rows, cols = 40, 256
    W = _weights(rng, rows, cols, zero_groups=False)
    bb = orc.rtn_quantize(W)
    prm = orc.params(C=64, P=4, b=4, S=64)
    cands = orc.encode_tiles(prm, W, bb["W0"], (rng.lognormal(0, 1, cols) ** 2).astype(np.float32))
    stream, counts, _ = orc.select_records(prm, [(rows, cols)], cands, [2.0])
    K = int(counts.sum())
    raw = np.frombuffer(stream, np.uint8).copy()
    h, T = orc.header_bytes(1), rows * cols // 64
    L = orc.record_bytes(prm, T)
    tb = int(np.ceil(np.log2(T)))
    rec = lambda k: int.from_bytes(raw[h + k * L: h + (k + 1) * L].tobytes(), "little")
    mask = (1 << tb) - 1
    dup = raw.copy()
    dup[h + L: h + 2 * L] = np.frombuffer(((rec(1) & ~mask) | (rec(0) & mask)).to_bytes(L, "little"), np.uint8)
    fixed = np.concatenate([raw[:h], dup[h + L:]])
    x = rng.normal(0, 1, (2, cols)).astype(np.float32)
    y, yabs, bad = orc.packed_gemv(prm, bb["q"], bb["s_eff"], 128, dup.tobytes(), K, x)
    yf, yabsf, badf = orc.packed_gemv(prm, bb["q"], bb["s_eff"], 128, fixed.tobytes(), K - 1, x)
    assert bad == 0 and badf == 0
    assert np.array_equal(y, yf) and np.array_equal(yabs, yabsf)
    y2, _, _ = orc.packed_gemv(prm, bb["q"], bb["s_eff"], 128, raw.tobytes(), K, x)
    assert not np.allclose(y, y2)


def test_packed_product_second_module_of_a_stream(orc):
    """Module 1 of a two-module stream: only its own records apply (tile
    offsets), matching the oracle decoder's weights of that module."""
    rng = np.random.default_rng(6)
    shapes = [(32, 256), (40, 384)]
    Ws = [_weights(rng, r, c, zero_groups=False) for r, c in shapes]
    bbs = [orc.rtn_quantize(W) for W in Ws]
    prm = orc.params(C=64, P=4, b=4, S=32)
    cands = np.concatenate([orc.encode_tiles(prm, W, bb["W0"], (rng.lognormal(0, 1, W.shape[1]) ** 2)
                                             .astype(np.float32)) for W, bb in zip(Ws, bbs)])
    stream, counts, _ = orc.select_records(prm, shapes, cands, [2.0])
    K = int(counts.sum())
    x = rng.normal(0, 1, (2, shapes[1][1])).astype(np.float32)
    y, yabs, bad = orc.packed_gemv(prm, bbs[1]["q"], bbs[1]["s_eff"], 128, stream, K, x, shapes=shapes, m=1)
    dec, _ = orc.decode_apply(prm, [bb["W0"] for bb in bbs], stream, K)
    ref = x.astype(np.float64) @ dec[1].astype(np.float64).T
    assert bad == 0 and counts[1] > 0
    assert (np.abs(y - ref) <= 2.0 ** -22 * yabs + 1e-30).all()
