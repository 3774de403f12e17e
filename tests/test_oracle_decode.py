"""Pins of the oracle's decoder (Sec. 3.2): an empty sidecar returns W0
exactly, tiles without a record are unchanged, the applied correction is
B_s * alpha_hat (double-precision reconstruction), the repaired tile's weighted
error reduction equals the encoder's gain (Eq. 4), and BF16 output is torch's
round-to-nearest-even of the float result."""
import numpy as np
import torch


def _setup(orc, rng, prm, shapes):
    mods, fis = [], []
    for rows, cols in shapes:
        W0 = rng.normal(0, 0.02, (rows, cols)).astype(np.float32)
        W = (W0 + rng.normal(0, 1e-3, (rows, cols))).astype(np.float32)
        act = rng.lognormal(0, 1.0, cols).astype(np.float32)
        mods.append((W, W0, act))
        fis.append(rng.lognormal(0, 1.5, (rows, cols)).astype(np.float32))
    if prm.variant == 1:
        cands = np.concatenate([orc.encode_tiles(prm, W, W0, a, fisher=F, w_act=0.5, w_fisher=0.5)
                                for (W, W0, a), F in zip(mods, fis)])
    else:
        cands = np.concatenate([orc.encode_tiles(prm, W, W0, a) for W, W0, a in mods])
    return mods, cands, fis


def test_empty_sidecar_returns_w0(orc):
    rng = np.random.default_rng(31)
    prm = orc.params(C=16, P=2, b=4, S=8)
    mods, cands, fis = _setup(orc, rng, prm, [(8, 32)])
    stream, counts, _ = orc.select_records(prm, [(8, 32)], cands, [4.0])
    outs, bad = orc.decode_apply(prm, [mods[0][1]], stream, 0)
    assert bad == 0 and np.array_equal(outs[0], mods[0][1])


def test_decode_reconstructs_encoder_correction(orc):
    rng = np.random.default_rng(32)
    for smode in (0, 1):
        prm = orc.params(C=16, P=4, b=4, S=16, scale_mode=smode, b_e=16 if smode else 8)
        shapes = [(16, 64), (8, 32)]
        mods, cands, fis = _setup(orc, rng, prm, shapes)
        stream, counts, _ = orc.select_records(prm, shapes, cands, [2.0])
        K = int(sum(counts))
        outs, bad = orc.decode_apply(prm, [m[1] for m in mods], stream, K)
        assert bad == 0
        T_m = [r * c // 16 for r, c in shapes]
        touched = [set() for _ in shapes]
        h = orc.header_bytes(2)
        L = orc.record_bytes(prm, sum(T_m))
        for k in range(K):
            t, c = orc.unpack_record(prm, sum(T_m), stream[h + k * L:h + (k + 1) * L])
            m = 0 if t < T_m[0] else 1
            lt = t - (0 if m == 0 else T_m[0])
            W, W0, act = mods[m]
            n_cb = W.shape[1] // 16
            i, cb = divmod(lt, n_cb)
            sl = slice(cb * 16, cb * 16 + 16)
            touched[m].add((i, cb))
            B = orc.basis_matrix(prm.gen_seed, int(c["seed"]), 16, 4)
            rhat = B @ (c["code"][:4].astype(np.float64) * orc.scale_value(prm, c["scale"]))
            got = outs[m][i, sl].astype(np.float64) - W0[i, sl]
            assert np.allclose(got, rhat, rtol=0, atol=4 * np.finfo(np.float32).eps * (np.abs(W0[i, sl]).max() + np.abs(rhat).max()))
            # Eq. 4 measured on the repaired weights equals the encoder's gain
            r = (W[i, sl] - W0[i, sl]).astype(np.float64)
            e = (W[i, sl] - outs[m][i, sl]).astype(np.float64)
            d = act[sl].astype(np.float64)
            g_dec = float(np.sum(d * (r * r - e * e)))
            energy = float(np.sum(d * r * r))
            assert abs(g_dec - cands[t]["gain"]) <= 2e-3 * energy
        for m, (W, W0, act) in enumerate(mods):
            n_cb = W.shape[1] // 16
            for i in range(W.shape[0]):
                for cb in range(n_cb):
                    if (i, cb) not in touched[m]:
                        sl = slice(cb * 16, cb * 16 + 16)
                        assert np.array_equal(outs[m][i, sl], W0[i, sl])


def test_prefix_decodes_without_refit(orc):
    rng = np.random.default_rng(33)
    prm = orc.params(C=16, P=4, b=4, S=8, variant=1)
    shapes = [(16, 64)]
    mods, cands, fis = _setup(orc, rng, prm, shapes)
    stream, counts, nbytes = orc.select_records(prm, shapes, cands, [1.0, 3.0])
    full, _ = orc.decode_apply(prm, [mods[0][1]], stream, int(counts[1]))
    pre, _ = orc.decode_apply(prm, [mods[0][1]], stream[:int(nbytes[0])], int(counts[0]))
    W, W0, act = mods[0]
    # error under the blended weights the progressive ranking uses (Sec. 3.3)
    dw = (np.float32(0.5) * act[None, :] + np.float32(0.5) * fis[0]).astype(np.float64)
    err = lambda What: float(np.sum(dw * (W - What.astype(np.float64)) ** 2))
    assert counts[0] < counts[1]
    assert err(full[0]) < err(pre[0]) < err(W0)


def test_bf16_output_rounding(orc):
    rng = np.random.default_rng(34)
    prm = orc.params(C=16, P=4, b=4, S=8)
    mods, cands, fis = _setup(orc, rng, prm, [(8, 64)])
    stream, counts, _ = orc.select_records(prm, [(8, 64)], cands, [4.0])
    f32, _ = orc.decode_apply(prm, [mods[0][1]], stream, int(counts[0]))
    b16, _ = orc.decode_apply(prm, [mods[0][1]], stream, int(counts[0]), out_bf16=True)
    ref = torch.from_numpy(f32[0]).to(torch.bfloat16).float().numpy()
    assert np.array_equal(b16[0], ref)
