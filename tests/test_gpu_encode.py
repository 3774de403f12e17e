"""GPU parity of the seed search (Sec. 3.2) against the oracle: every candidate
field bit for bit, over the specialised (C=64, P=4, U) kernel and the generic
kernel, both variants, both scale modes, ragged rows and seed counts, seed
splits, and the degenerate tiles."""
import numpy as np
import pytest
import torch

from gpu_util import assert_candidates_equal, oracle_encode, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def aw():
    import paper_2608_23144_gb300 as aw
    assert torch.cuda.is_available()
    return aw


def _mods(shapes, w_dtype="bf16", fisher=False, seed=0, blend=(0.5, 0.5)):
    from synth import make_module
    return [make_module(r, c, seed=seed + 17 * i, device="cpu", w_dtype=w_dtype, fisher=fisher, blend=blend)
            for i, (r, c) in enumerate(shapes)]


CASES = [
    # (label, params, shapes, w_dtype, fisher)
    ("c64p4_u_pow2", dict(C=64, P=4, b=4, S=96), [(200, 256), (64, 128), (1, 64)], "bf16", False),
    ("c64p4_u_fp16_single_256x512", dict(C=64, P=4, b=4, S=256, scale_mode=1, b_e=16), [(256, 512)], "f32", False),
    ("c64p4_u_ridge0_nopermute", dict(C=64, P=4, b=4, S=40, ridge_rel=0.0, permute=0), [(130, 192)], "bf16", False),
    ("c64p4_pf", dict(C=64, P=4, b=4, S=48, variant=1), [(70, 128), (33, 64)], "bf16", True),
    ("c16p4_pf_paper", dict(C=16, P=4, b=4, S=16, variant=1), [(96, 64), (40, 48)], "bf16", True),
    ("c128p2_u_paper", dict(C=128, P=2, b=4, S=2), [(64, 256), (17, 128)], "bf16", False),
    ("c8p2_b3_u", dict(C=8, P=2, b=3, S=33), [(50, 24)], "f32", False),
    ("c32p3_b2_u_ebias", dict(C=32, P=3, b=2, S=20, b_e=5, e_bias=-12), [(45, 96)], "bf16", False),
    ("c256p8_b8_u", dict(C=256, P=8, b=8, S=12), [(20, 512)], "bf16", False),
    ("c4p1_u", dict(C=4, P=1, b=4, S=9), [(11, 20)], "f32", False),
    ("c64p4_u_fp16_pf", dict(C=64, P=4, b=4, S=24, variant=1, scale_mode=1, b_e=16), [(40, 128)], "f32", True),
    ("c64p3_u_generic", dict(C=64, P=3, b=4, S=70), [(90, 192), (5, 64)], "bf16", False),
    ("c64p2_pf_generic", dict(C=64, P=2, b=3, S=21, variant=1), [(77, 128)], "bf16", True),
    ("c32p4_pf_s3", dict(C=32, P=4, b=4, S=3, variant=1), [(50, 96)], "f32", True),
    # the tcgen05 P_F search takes 12-seed chunks: selectors padded to 96
    ("c64p4_pf_s100", dict(C=64, P=4, b=4, S=100, variant=1), [(140, 192), (3, 64)], "bf16", True),
    ("c64p4_pf_s13_b5", dict(C=64, P=4, b=5, S=13, variant=1), [(33, 128)], "f32", True),
]


@pytest.mark.parametrize("label,kw,shapes,w_dtype,fisher", CASES, ids=[c[0] for c in CASES])
def test_encode_matches_oracle(aw, orc, label, kw, shapes, w_dtype, fisher):
    mods = _mods(shapes, w_dtype, fisher)
    prm, oprm = aw.params(**kw), orc.params(**kw)
    cands = aw.awsrc_encode_tiles(prm, to_dev(mods))
    flags = aw.awsrc_workspace_status(cands._awsrc_workspace)
    got = aw.candidates_to_numpy(cands)
    want = np.concatenate(oracle_encode(orc, oprm, mods))
    assert flags == 0, f"device fault flags {flags:#x}"
    assert_candidates_equal(got, want, label)
    assert np.isfinite(got["gain"]).sum() > 0.5 * len(got)


@pytest.mark.parametrize("kind", ["wide_range", "sparse_weights", "large_ridge", "one_hot_residual"])
def test_pruned_search_matches_oracle_on_adversarial_tiles(aw, orc, kind):
    """The specialised search skips candidates whose gain bound cannot beat the
    running best. On tiles built to stress that bound (activation moments over
    twelve decades, mostly-zero weights that make G singular, a large ridge,
    one-hot residuals with many equal correlations) the winners must still be
    the oracle's, bit for bit."""
    mods = _mods([(300, 256)], "bf16", seed=3)
    m = mods[0]
    g = torch.Generator().manual_seed(7)
    kw = dict(C=64, P=4, b=4, S=512)
    if kind == "wide_range":
        m["act"] = (10.0 ** (torch.rand(256, generator=g) * 12 - 6)).float()
    elif kind == "sparse_weights":
        m["act"] = m["act"] * (torch.rand(256, generator=g) < 0.1).float()
    elif kind == "large_ridge":
        kw["ridge_rel"] = 0.5
    else:
        W = m["W0"].clone()
        W[:, ::64] += 0.25
        m["W"] = W
    prm, oprm = aw.params(**kw), orc.params(**kw)
    cands = aw.awsrc_encode_tiles(prm, to_dev(mods))
    flags = aw.awsrc_workspace_status(cands._awsrc_workspace)
    got = aw.candidates_to_numpy(cands)
    want = oracle_encode(orc, oprm, mods)[0]
    assert flags == 0, f"device fault flags {flags:#x}"
    assert_candidates_equal(got, want, kind)


@pytest.mark.parametrize("kind", ["wide_fisher", "sparse_fisher", "sparse_ridge0", "tiny_sparse_ridge0"])
def test_pf_search_matches_oracle_on_adversarial_weights(aw, orc, kind):
    """The tcgen05 P_F search takes the fast reciprocal of a pivot only while
    every pivot of the warp's two seed pairs is in [2^-125, 2^125); otherwise
    it takes the exact validity checks and correctly rounded reciprocals.
    Fisher weights over twelve decades; mostly-zero Fisher weights with no
    activation part (singular Gram matrices held off by the ridge alone, or,
    without a ridge, pivots of zero, rounding residue or either sign, which
    take the exact branch); and the same near the smallest element weights the
    fixed-point grids take (1e-28): the oracle's candidates bit for bit."""
    sparse = kind != "wide_fisher"
    mods = _mods([(130, 192), (7, 64)], "bf16", fisher=True, seed=11, blend=(0.0, 1.0) if sparse else (0.5, 0.5))
    g = torch.Generator().manual_seed(13)
    for m in mods:
        F = m["fisher"]
        if sparse:
            F = F * (torch.rand(F.shape, generator=g) < 0.1).float()
        else:
            F = F * (10.0 ** (torch.rand(F.shape, generator=g) * 12 - 6)).float()
        if kind == "tiny_sparse_ridge0":
            F = F * 1e-29
        m["fisher"] = F
    kw = dict(C=64, P=4, b=4, S=48, variant=1)
    if kind.endswith("ridge0"):
        kw["ridge_rel"] = 0.0
    prm, oprm = aw.params(**kw), orc.params(**kw)
    cands = aw.awsrc_encode_tiles(prm, to_dev(mods))
    flags = aw.awsrc_workspace_status(cands._awsrc_workspace)
    got = aw.candidates_to_numpy(cands)
    want = np.concatenate(oracle_encode(orc, oprm, mods))
    assert flags == 0, f"device fault flags {flags:#x}"
    assert_candidates_equal(got, want, kind)
    assert np.isfinite(want["gain"]).sum() > 0, "no tile with a valid candidate"


@pytest.mark.parametrize("variant", [0, 1])
def test_padding_selectors_never_win(aw, orc, variant):
    """Seeds are searched in chunks padded up to a multiple of 32 with all-zero
    masks; such a basis is four copies of the constant vector, which would fit a
    constant residual exactly. The padding must never be chosen."""
    mods = _mods([(64, 128)], "f32", fisher=bool(variant), seed=5)
    m = mods[0]
    m["W"] = m["W0"] + 0.01                          # constant residual on every tile
    m["W"][::3, :64] += 0.002 * torch.randn(22, 64)  # and some ordinary tiles
    kw = dict(C=64, P=4, b=4, S=37, variant=variant)
    prm, oprm = aw.params(**kw), orc.params(**kw)
    cands = aw.awsrc_encode_tiles(prm, to_dev(mods))
    flags = aw.awsrc_workspace_status(cands._awsrc_workspace)
    got = aw.candidates_to_numpy(cands)
    want = oracle_encode(orc, oprm, mods)[0]
    assert flags == 0, f"device fault flags {flags:#x}"
    assert (got["seed"] < 37).all()
    assert_candidates_equal(got, want, f"padding v{variant}")


def test_degenerate_tiles(aw, orc):
    mods = _mods([(40, 192)], "f32")
    m = mods[0]
    m["W"][0, :64] = m["W0"][0, :64]          # zero residual tile
    m["act"][64:128] = 0.0                   # zero-weight column block (every row)
    m["W"][3, 130] = 1e6                     # residual outside the supported domain
    m["W"][5, 10] = float("nan")             # non-finite residual
    m["act"][150] = float("inf")             # non-finite activation moment
    prm, oprm = aw.params(C=64, P=4, S=64), orc.params(C=64, P=4, S=64)
    got = aw.candidates_to_numpy(aw.awsrc_encode_tiles(prm, to_dev(mods)))
    want = oracle_encode(orc, oprm, mods)[0]
    assert_candidates_equal(got, want, "degenerate")
    n_cb = 3
    for t in [0, 3 * n_cb + 2, 5 * n_cb + 0] + [i * n_cb + 1 for i in range(40)] + [i * n_cb + 2 for i in range(40)]:
        assert got["gain"][t] == -np.inf and got["seed"][t] == 0 and not got["code"][t].any()


@pytest.mark.parametrize("variant", [0, 1])
def test_seed_splits_do_not_change_the_result(aw, orc, variant):
    """A small module is split over many blocks along the seed axis; a large one is
    not. The same rows embedded in both must give identical candidates."""
    mods = _mods([(8, 64)], "bf16", fisher=bool(variant))
    big = _mods([(1500, 64)], "bf16", seed=5, fisher=bool(variant))
    big[0]["W"][:8] = mods[0]["W"]
    big[0]["W0"][:8] = mods[0]["W0"]
    big[0]["act"] = mods[0]["act"].clone()
    if variant:
        big[0]["fisher"][:8] = mods[0]["fisher"]
        big[0]["w_act"], big[0]["w_fisher"] = mods[0]["w_act"], mods[0]["w_fisher"]
    prm = aw.params(C=64, P=4, S=512, variant=variant)
    a = aw.candidates_to_numpy(aw.awsrc_encode_tiles(prm, to_dev(mods)))
    b = aw.candidates_to_numpy(aw.awsrc_encode_tiles(prm, to_dev(big)))[:8]
    assert_candidates_equal(a, b, "split vs unsplit")


def test_gen_basis_matches_oracle(aw, orc):
    """Every selector's masks, bit for bit (C <= 64 takes the warp-parallel
    Fisher-Yates evaluation, C > 64 the sequential one)."""
    cases = [(64, 4, 1, 4096), (64, 8, 1, 300), (64, 4, 0, 100), (32, 4, 1, 500), (16, 4, 1, 64), (8, 3, 1, 100),
             (4, 2, 1, 200), (4, 4, 1, 64), (4, 1, 0, 8), (128, 2, 1, 64), (256, 8, 0, 32), (256, 4, 1, 40)]
    for C, P, permute, S in cases:
        prm = aw.params(C=C, P=P, S=S, permute=permute, gen_seed=12345)
        W = (C + 63) // 64
        masks = aw.awsrc_gen_basis(prm).cpu().numpy().view(np.uint64).reshape(S, P, W)
        bits = ((masks[..., None] >> np.arange(64, dtype=np.uint64)) & np.uint64(1)).astype(np.uint8)
        bits = bits.reshape(S, P, W * 64)
        assert not bits[:, :, C:].any(), (C, P)
        for s in range(S):
            neg = orc.gen_basis(12345, s, C, P, permute)[3]
            assert np.array_equal(bits[s, :, :C], neg), (C, P, permute, s)


