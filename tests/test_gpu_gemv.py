"""GPU parity of the packed product y = (W0 + r_hat) x (sidecar applied inside
an INT4 product, W_hat never formed) against the oracle's double-precision
definition, within the binary32 summation bound the header states; streams are
the oracle's own (encode and select on the CPU), the packed backbone is the
GPU's (bit-identical to the oracle's, tests/test_gpu_backbone.py)."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def aw():
    import paper_2608_23144_gb300 as aw
    assert torch.cuda.is_available()
    return aw


def _weights(rng, rows, cols):
    W = rng.normal(0, 0.02, (rows, cols)).astype(np.float32)
    W[:, rng.choice(cols, max(1, cols // 100), replace=False)] *= 8.0
    return W


def _bound(cols, C, yabs):
    """The header's bound: (cols / min(C, 32) + 32) * 2^-24 * sum_j (|W0 x| + |r x|)."""
    return (cols / min(C, 32) + 32) * 2.0 ** -24 * yabs + 1e-30


@pytest.mark.parametrize("sdq", [False, True])
@pytest.mark.parametrize("kw", [dict(C=64, P=4, b=4, S=64), dict(C=16, P=4, b=4, S=16, scale_mode=1, b_e=16),
                                dict(C=32, P=4, b=5, S=32), dict(C=64, P=4, b=6, S=32),
                                dict(C=8, P=4, b=3, S=16),
                                dict(C=128, P=2, b=4, S=8)])
def test_packed_gemv_matches_definition(aw, orc, sdq, kw):
    rng = np.random.default_rng(11)
    shapes = [(96, 512), (70, 384)]
    Ws = [_weights(rng, r, c) for r, c in shapes]
    obb = [orc.rtn_quantize(W, sdq=sdq) for W in Ws]
    oprm, prm = orc.params(**kw), aw.params(**kw)
    cands = np.concatenate([orc.encode_tiles(oprm, W, bb["W0"], (rng.lognormal(0, 1, W.shape[1]) ** 2)
                                             .astype(np.float32)) for W, bb in zip(Ws, obb)])
    stream, counts, _ = orc.select_records(oprm, shapes, cands, [2.0])
    K = int(counts.sum())
    assert counts.min() > 0
    side = aw.awsrc_sidecar_prepare(prm, shapes, torch.from_numpy(np.frombuffer(stream, np.uint8).copy()).cuda(), K)
    assert aw.awsrc_workspace_status(side) == 0
    for m, (rows, cols) in enumerate(shapes):
        bb = aw.awsrc_rtn_quantize(torch.from_numpy(Ws[m]).cuda(), sdq=sdq)
        for M in (1, 3, 8):
            x = rng.normal(0, 1, (M, cols)).astype(np.float32)
            xd = torch.from_numpy(x).cuda()
            y = aw.awsrc_packed_gemv(prm, shapes, m, bb, xd, sidecar=side).cpu().numpy()
            want, yabs, bad = orc.packed_gemv(oprm, obb[m]["q"], obb[m]["s_eff"], 128, stream, K, x,
                                              shapes=shapes, m=m)
            assert bad == 0
            assert (np.abs(y - want) <= _bound(cols, kw["C"], yabs)).all(), (m, M)
            # no sidecar: the backbone alone
            y0 = aw.awsrc_packed_gemv(prm, shapes, m, bb, xd).cpu().numpy()
            want0, yabs0, _ = orc.packed_gemv(oprm, obb[m]["q"], obb[m]["s_eff"], 128, stream, 0, x,
                                              shapes=shapes, m=m)
            assert (np.abs(y0 - want0) <= _bound(cols, kw["C"], yabs0)).all()
            assert not np.allclose(y, y0)


def test_packed_gemv_full_size_down_projection(aw, orc):
    """A Qwen2.5-3B down projection (2048 x 11008) with SDQ, one vector, a
    0.162-bit/weight stream from the library's own encoder and selector (the
    oracle checks the product from that stream and its own backbone)."""
    rng = np.random.default_rng(12)
    rows, cols = 2048, 11008
    W = _weights(rng, rows, cols)
    obb = orc.rtn_quantize(W, sdq=True)
    kw = dict(C=64, P=4, b=4, S=256)
    prm, oprm = aw.params(**kw), orc.params(**kw)
    Wd = torch.from_numpy(W).cuda()
    bb = aw.awsrc_rtn_quantize(Wd, sdq=True)
    act = torch.from_numpy((rng.lognormal(0, 1, cols) ** 2).astype(np.float32)).cuda()
    mods = [{"W": Wd, "W0": bb["W0"], "act": act}]
    cands = aw.awsrc_encode_tiles(prm, mods)
    stream, counts, nbytes = aw.awsrc_select_records(prm, mods, cands, [0.162])
    K = int(counts.sum())
    side = aw.awsrc_sidecar_prepare(prm, [(rows, cols)], stream, K)
    x = rng.normal(0, 1, (1, cols)).astype(np.float32)
    y = aw.awsrc_packed_gemv(prm, [(rows, cols)], 0, bb, torch.from_numpy(x).cuda(), sidecar=side).cpu().numpy()
    host_stream = bytes(stream.cpu().numpy()[: int(nbytes[0])])
    want, yabs, bad = orc.packed_gemv(oprm, obb["q"], obb["s_eff"], 128, host_stream, K, x)
    assert bad == 0 and K > 10000
    assert (np.abs(y - want) <= _bound(cols, 64, yabs)).all()


@pytest.mark.parametrize("M", [1, 3, 8])
def test_packed_gemv_batch_equals_single_calls(aw, orc, M):
    """One launch for several (module, x) tasks, modules repeated and x shared
    (as q/k/v share their input): every y is bit-identical to its single call
    and within the bound of the definition. With M = 8 the 4096-column module's
    inputs exceed shared memory and take their own launch."""
    rng = np.random.default_rng(13)
    shapes = [(96, 512), (40, 4096), (130, 1024)]
    kw = dict(C=64, P=4, b=4, S=64)
    oprm, prm = orc.params(**kw), aw.params(**kw)
    Ws = [_weights(rng, r, c) for r, c in shapes]
    obb = [orc.rtn_quantize(W, sdq=True) for W in Ws]
    cands = np.concatenate([orc.encode_tiles(oprm, W, bb["W0"], (rng.lognormal(0, 1, W.shape[1]) ** 2)
                                             .astype(np.float32)) for W, bb in zip(Ws, obb)])
    stream, counts, _ = orc.select_records(oprm, shapes, cands, [1.0])
    K = int(counts.sum())
    assert counts.min() > 0
    side = aw.awsrc_sidecar_prepare(prm, shapes, torch.from_numpy(np.frombuffer(stream, np.uint8).copy()).cuda(), K)
    bbs = [aw.awsrc_rtn_quantize(torch.from_numpy(W).cuda(), sdq=True) for W in Ws]
    xs = [torch.from_numpy(rng.normal(0, 1, (M, c)).astype(np.float32)).cuda() for _, c in shapes]
    x0b = torch.from_numpy(rng.normal(0, 1, (M, shapes[0][1])).astype(np.float32)).cuda()
    tasks = [(0, bbs[0], xs[0]), (2, bbs[2], xs[2]), (1, bbs[1], xs[1]), (0, bbs[0], x0b), (0, bbs[0], xs[0])]
    ys = aw.awsrc_packed_gemv_batch(prm, shapes, tasks, sidecar=side)
    for (m, bb, x), y in zip(tasks, ys):
        single = aw.awsrc_packed_gemv(prm, shapes, m, bb, x, sidecar=side)
        assert torch.equal(y, single), m
        want, yabs, bad = orc.packed_gemv(oprm, obb[m]["q"], obb[m]["s_eff"], 128, stream, K, x.cpu().numpy(),
                                          shapes=shapes, m=m)
        assert bad == 0
        assert (np.abs(y.cpu().numpy() - want) <= _bound(shapes[m][1], 64, yabs)).all(), m
    assert torch.equal(ys[0], ys[4]) and not torch.equal(ys[0], ys[3])
