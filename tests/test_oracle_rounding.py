"""Pins of the oracle's binary16 / bfloat16 conversions and of c = RN(C^-1/2)
against numpy and torch (independent implementations of IEEE rounding)."""
import numpy as np
import torch


def _edge_values():
    rng = np.random.default_rng(3)
    vals = [0.0, -0.0, 1.0, -1.0, 65504.0, 65519.99, 65520.0, 1e6, 6.1035156e-05, 6.0e-05,
            5.9604645e-08, 2.98e-08, 2.9802322e-08, 3.0e-08, 1e-10, 0.1, 1 / 3, np.float32(1e-4) * 1.4]
    vals += list(rng.normal(0, 1, 2000)) + list(rng.lognormal(-10, 6, 4000) * rng.choice([-1, 1], 4000))
    # exact binary16 midpoints (ties) in the normal and subnormal ranges
    h = rng.integers(1, 0x7bff, 2000).astype(np.uint16)
    lo = h.view(np.float16).astype(np.float32)
    hi = (h + 1).view(np.float16).astype(np.float32)
    vals += list(((lo.astype(np.float64) + hi.astype(np.float64)) / 2).astype(np.float32))
    return np.array(vals, np.float32)


def test_f32_to_f16_matches_numpy(orc):
    v = _edge_values()
    ref = v.astype(np.float16).view(np.uint16)
    got = np.array([orc.f32_to_f16_bits(float(x)) for x in v], np.uint16)
    assert np.array_equal(got, ref)
    back = np.array([orc.f16_bits_to_f32(int(h)) for h in ref], np.float32)
    assert np.array_equal(back, ref.view(np.float16).astype(np.float32))


def test_f32_to_bf16_matches_torch(orc):
    v = _edge_values()
    ref = torch.from_numpy(v).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = np.array([orc.f32_to_bf16_bits(float(x)) for x in v], np.uint16)
    assert np.array_equal(got, ref)


def test_basis_normaliser_is_correctly_rounded(orc):
    # the oracle's decoder and fit use c = RN(C^-1/2); check through a d = 1 tile
    for C in (4, 8, 16, 32, 64, 128, 256):
        prm = orc.params(C=C, P=1, b=8, S=1, ridge_rel=0.0)
        r = np.zeros(C, np.float32)
        neg = orc.gen_basis(0, 0, C, 1, 1)[3]
        # put r = +1 on the first coordinate with the basis sign: u = 1, b = c, alpha = c
        r[0] = -1.0 if neg[0, 0] else 1.0
        out = orc.score_candidate(prm, r, np.ones(C, np.float32), neg)
        assert out["alpha"][0] == np.float32(1.0 / np.sqrt(np.float64(C)))
