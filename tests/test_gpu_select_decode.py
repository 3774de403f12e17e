"""GPU parity of selection/serialisation (Sec. 3.3-3.4, Eq. 5) and of the
decoder (Sec. 3.2): stream bytes, counts and byte totals identical to the
oracle's; repaired weights identical element by element in every mode."""
import numpy as np
import pytest
import torch

from gpu_util import oracle_encode, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def aw():
    import paper_2608_23144_gb300 as aw
    return aw


def _setup(aw, orc, shapes, kw, w_dtype="bf16", fisher=False, seed=3):
    from synth import make_module
    mods = [make_module(r, c, seed=seed + 7 * i, device="cpu", w_dtype=w_dtype, fisher=fisher,
                        blend=(0.5, 0.5)) for i, (r, c) in enumerate(shapes)]
    prm, oprm = aw.params(**kw), orc.params(**kw)
    dmods = to_dev(mods)
    cands = aw.awsrc_encode_tiles(prm, dmods)
    ocands = np.concatenate(oracle_encode(orc, oprm, mods))
    assert np.array_equal(aw.candidates_to_numpy(cands).view(np.uint8), ocands.view(np.uint8))
    return mods, dmods, prm, oprm, cands, ocands


@pytest.mark.parametrize("rate", [0.162, 0.5, 2.0])
def test_select_u_matches_oracle(aw, orc, rate):
    shapes = [(200, 256), (64, 128), (33, 64), (128, 512)]
    mods, dmods, prm, oprm, cands, ocands = _setup(aw, orc, shapes, dict(C=64, P=4, b=4, S=64))
    stream, counts, nbytes = aw.awsrc_select_records(prm, dmods, cands, [rate])
    ostream, ocounts, obytes = orc.select_records(oprm, shapes, ocands, [rate])
    assert list(counts.cpu().numpy()) == list(ocounts)
    assert list(nbytes.cpu().numpy()) == list(obytes)
    assert bytes(stream.cpu().numpy()[: int(nbytes[0])]) == ostream


def test_select_pf_prefixes_match_oracle(aw, orc):
    shapes = [(96, 64), (40, 48), (64, 128)]
    mods, dmods, prm, oprm, cands, ocands = _setup(aw, orc, shapes, dict(C=16, P=4, b=4, S=16, variant=1),
                                                   fisher=True)
    rates = [0.05, 0.10, 0.162, 0.25, 3.0]
    stream, counts, nbytes = aw.awsrc_select_records(prm, dmods, cands, rates)
    ostream, ocounts, obytes = orc.select_records(oprm, shapes, ocands, rates)
    assert list(counts.cpu().numpy()) == list(ocounts)
    assert list(nbytes.cpu().numpy()) == list(obytes)
    assert bytes(stream.cpu().numpy()[: int(nbytes.max())]) == ostream


def test_select_many_modules_and_ties(aw, orc):
    """40 modules (module index takes 6 key bits) and candidates with exactly equal
    gains: ties are broken by tile index in both implementations."""
    shapes = [(8 + (i % 5), 64) for i in range(40)]
    mods, dmods, prm, oprm, cands, ocands = _setup(aw, orc, shapes, dict(C=64, P=4, b=4, S=32))
    c = aw.candidates_to_numpy(cands).copy()
    c["gain"][::3] = np.float32(1e-5)      # force ties
    c["gain"][1::7] = -np.inf
    c["gain"][2::11] = 0.0
    dc = torch.from_numpy(c.view(np.uint8).reshape(-1, 16).copy()).cuda()
    for prm_, oprm_ in [(prm, oprm), (aw.params(C=64, P=4, b=4, S=32, variant=1),
                                      orc.params(C=64, P=4, b=4, S=32, variant=1))]:
        rates = [1.0] if prm_.variant == 0 else [0.3, 1.0]
        stream, counts, nbytes = aw.awsrc_select_records(prm_, dmods, dc, rates)
        ostream, ocounts, obytes = orc.select_records(oprm_, shapes, c, rates)
        assert list(counts.cpu().numpy()) == list(ocounts)
        assert bytes(stream.cpu().numpy()[: int(nbytes.max())]) == ostream


@pytest.mark.parametrize("w_dtype,out_dtype", [("bf16", torch.bfloat16), ("f32", torch.float32),
                                               ("f32", torch.bfloat16), ("bf16", torch.float32)])
def test_decode_dense_matches_oracle(aw, orc, w_dtype, out_dtype):
    shapes = [(100, 256), (64, 128)]
    kw = dict(C=64, P=4, b=4, S=64, scale_mode=1, b_e=16) if w_dtype == "f32" else dict(C=64, P=4, b=4, S=64)
    mods, dmods, prm, oprm, cands, ocands = _setup(aw, orc, shapes, kw, w_dtype=w_dtype)
    stream, counts, nbytes = aw.awsrc_select_records(prm, dmods, cands, [1.0])
    ostream, ocounts, _ = orc.select_records(oprm, shapes, ocands, [1.0])
    K = int(ocounts.sum())
    W0s = [m["W0"].float().numpy() for m in mods]
    for k in (0, K // 3, K, -1):
        outs = aw.awsrc_decode_apply(prm, dmods, stream, k, out_dtype=out_dtype)
        torch.cuda.synchronize()
        oouts, _ = orc.decode_apply(oprm, W0s, ostream, K if k < 0 else k,
                                    out_bf16=(out_dtype == torch.bfloat16))
        for g, o in zip(outs, oouts):
            assert np.array_equal(g.float().cpu().numpy(), o), k
        assert aw.awsrc_workspace_status(outs[0]._awsrc_workspace) == 0


def test_decode_inplace_matches_dense(aw, orc):
    shapes = [(100, 256), (64, 128), (10, 64)]
    mods, dmods, prm, oprm, cands, ocands = _setup(aw, orc, shapes, dict(C=64, P=4, b=4, S=64))
    stream, counts, nbytes = aw.awsrc_select_records(prm, dmods, cands, [1.0])
    K = int(counts.sum())
    dense = aw.awsrc_decode_apply(prm, dmods, stream, K)
    inplace = [m["W0"].clone() for m in dmods]
    aw.awsrc_decode_apply(prm, dmods, stream, K, outs=inplace, mode=aw.DECODE_INPLACE)
    for a, b in zip(dense, inplace):
        assert torch.equal(a, b)
    # decoding against W0 itself (aliasing) gives the same weights
    alias = [{**m, "W0": m["W0"].clone()} for m in dmods]
    aw.awsrc_decode_apply(prm, alias, stream, K, outs=[m["W0"] for m in alias], mode=aw.DECODE_INPLACE)
    for a, m in zip(dense, alias):
        assert torch.equal(a, m["W0"])


def test_decode_skips_and_flags_out_of_range_records(aw, orc):
    """A stream written with S = 64 read back with S = 33: the seed field keeps its
    6-bit width, so records naming seeds 33..63 are out of range. They must be
    skipped (their tiles keep W0) and reported; the others are applied."""
    shapes = [(64, 128)]
    mods, dmods, prm, oprm, cands, ocands = _setup(aw, orc, shapes, dict(C=64, P=4, b=4, S=64))
    stream, counts, nbytes = aw.awsrc_select_records(prm, dmods, cands, [1.0])
    K = int(counts.sum())
    small, osmall = aw.params(C=64, P=4, b=4, S=33), orc.params(C=64, P=4, b=4, S=33)
    outs = aw.awsrc_decode_apply(small, dmods, stream, K)
    flags = aw.awsrc_workspace_status(outs[0]._awsrc_workspace)
    ostream = bytes(stream.cpu().numpy()[: int(nbytes[0])])
    oouts, obad = orc.decode_apply(osmall, [mods[0]["W0"].float().numpy()], ostream, K, out_bf16=True)
    assert obad == 1 and flags & 1, "out-of-range records must be reported"
    assert np.array_equal(outs[0].float().cpu().numpy(), oouts[0])


def test_decode_rejects_K_beyond_stream(aw, orc):
    shapes = [(64, 128)]
    mods, dmods, prm, oprm, cands, ocands = _setup(aw, orc, shapes, dict(C=64, P=4, b=4, S=64))
    stream, counts, nbytes = aw.awsrc_select_records(prm, dmods, cands, [1.0])
    with pytest.raises(aw.AwsrcError):
        aw.awsrc_decode_apply(prm, dmods, stream[: int(nbytes[0])], int(counts.sum()) + 1)


def test_decode_repeated_tile_takes_later_record(aw, orc):
    """A stream that names a tile twice (never written by the encoder) is reported;
    dense and in-place decoding apply the later record, i.e. they equal decoding
    the stream without the earlier one."""
    shapes = [(100, 256)]
    mods, dmods, prm, oprm, cands, ocands = _setup(aw, orc, shapes, dict(C=64, P=4, b=4, S=64))
    stream, counts, nbytes = aw.awsrc_select_records(prm, dmods, cands, [1.0])
    K = int(counts.sum())
    raw = stream.cpu().numpy()[: int(nbytes[0])].copy()
    h, T = orc.header_bytes(1), 100 * 256 // 64
    L = orc.record_bytes(oprm, T)
    tb = int(np.ceil(np.log2(T)))
    rec = lambda k: int.from_bytes(raw[h + k * L: h + (k + 1) * L].tobytes(), "little")
    mask = (1 << tb) - 1
    r1 = (rec(1) & ~mask) | (rec(0) & mask)        # record 1's payload on record 0's tile
    dup = raw.copy()
    dup[h + L: h + 2 * L] = np.frombuffer(r1.to_bytes(L, "little"), np.uint8)
    fixed = np.concatenate([raw[:h], dup[h + L:]])  # record 0 removed
    outs = aw.awsrc_decode_apply(prm, dmods, torch.from_numpy(dup).cuda(), K)
    flags = aw.awsrc_workspace_status(outs[0]._awsrc_workspace)
    assert flags & 1, "a repeated tile must be reported"
    oouts, obad = orc.decode_apply(oprm, [mods[0]["W0"].float().numpy()], fixed.tobytes(), K - 1, out_bf16=True)
    assert obad == 0
    assert np.array_equal(outs[0].float().cpu().numpy(), oouts[0])
    # in place (W_hat is W0 itself): the same result and the same report, on
    # every repetition (the later record claims the tile before any patch runs)
    for _ in range(3):
        w = dmods[0]["W0"].clone()
        out = aw.awsrc_decode_apply(prm, [{**dmods[0], "W0": w}], torch.from_numpy(dup).cuda(), K, outs=[w],
                                    mode=aw.DECODE_INPLACE)
        flags = aw.awsrc_workspace_status(out[0]._awsrc_workspace)
        assert flags & 1, "a repeated tile must be reported in place too"
        assert np.array_equal(w.float().cpu().numpy(), oouts[0])


@pytest.mark.parametrize("C,P", [(16, 4), (32, 4), (8, 2), (4, 1)])
def test_decode_dense_many_modules_small_tiles(aw, orc, C, P):
    """20 modules (two launch runs of at most 16) and tiles of one or two 16-byte
    vectors (and a 4-element tile, below one BF16 vector)."""
    shapes = [(6 + (i % 4), 32 if i % 3 else 64) for i in range(20)]
    kw = dict(C=C, P=P, b=4, S=16)
    mods, dmods, prm, oprm, cands, ocands = _setup(aw, orc, shapes, kw)
    stream, counts, nbytes = aw.awsrc_select_records(prm, dmods, cands, [2.0])
    ostream, ocounts, _ = orc.select_records(oprm, shapes, ocands, [2.0])
    K = int(ocounts.sum())
    assert K > 0
    outs = aw.awsrc_decode_apply(prm, dmods, stream, -1)
    oouts, _ = orc.decode_apply(oprm, [m["W0"].float().numpy() for m in mods], ostream, K, out_bf16=True)
    for g, o in zip(outs, oouts):
        assert np.array_equal(g.float().cpu().numpy(), o)
    assert aw.awsrc_workspace_status(outs[0]._awsrc_workspace) == 0


def test_clipping_exponent_field_with_bias(aw, orc):
    """A 3-bit exponent field with e_bias = -10 holds e in [-14, -7]: tiles whose
    coefficients need a larger exponent get -7 with their codes clamped to
    [-qmax, qmax] (the tcgen05 search without pruning), and the stream stores
    e - e_bias in 3 bits (2 e_bias is not a multiple of 8, so a bias applied
    with the wrong sign would change the bytes). Candidates, stream bytes and
    decoded weights match the oracle bit for bit."""
    shapes = [(100, 256), (64, 128)]
    mods, dmods, prm, oprm, cands, ocands = _setup(aw, orc, shapes, dict(C=64, P=4, b=4, S=64, b_e=3, e_bias=-10))
    assert (ocands["scale"][ocands["gain"] > -np.inf] == -7).sum() > 0    # the top of the field is reached
    stream, counts, nbytes = aw.awsrc_select_records(prm, dmods, cands, [1.0])
    ostream, ocounts, obytes = orc.select_records(oprm, shapes, ocands, [1.0])
    assert list(counts.cpu().numpy()) == list(ocounts)
    assert list(nbytes.cpu().numpy()) == list(obytes)
    assert bytes(stream.cpu().numpy()[: int(nbytes[0])]) == ostream
    K = int(ocounts.sum())
    W0s = [m["W0"].float().numpy() for m in mods]
    outs = aw.awsrc_decode_apply(prm, dmods, stream, K)
    torch.cuda.synchronize()
    oouts, _ = orc.decode_apply(oprm, W0s, ostream, K, out_bf16=True)
    for g, o in zip(outs, oouts):
        assert np.array_equal(g.float().cpu().numpy(), o)
    assert aw.awsrc_workspace_status(outs[0]._awsrc_workspace) == 0
