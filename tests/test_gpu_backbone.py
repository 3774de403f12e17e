"""GPU parity of the RTN-INT4 backbone and its scale double quantisation
(Eq. 1, Sec. 3.3, Sec. 4) against the oracle: packed codes, binary16 scales,
SDQ codes and constants and W0, bit for bit, over input and output dtypes,
partial SDQ blocks, zero groups and a full Qwen2.5-3B-sized gate projection."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def aw():
    import paper_2608_23144_gb300 as aw
    assert torch.cuda.is_available()
    return aw


def _weights(seed, rows, cols):
    rng = np.random.default_rng(seed)
    W = rng.normal(0, 0.02, (rows, cols)).astype(np.float32)
    W[:, rng.choice(cols, max(1, cols // 100), replace=False)] *= 8.0
    W[0, :128] = 0.0
    W[-1, -128:] *= 1e-3
    return W


def _pack(q):
    q = q.reshape(-1).astype(np.int16) & 15
    return (q[0::2] | (q[1::2] << 4)).astype(np.uint8)


@pytest.mark.parametrize("rows,cols", [(40, 512), (300, 1024), (11008, 2048)])
@pytest.mark.parametrize("w_dtype,w0_dtype", [(torch.bfloat16, torch.bfloat16), (torch.float32, torch.float32),
                                              (torch.bfloat16, torch.float32)])
@pytest.mark.parametrize("sdq", [False, True])
def test_backbone_matches_oracle(aw, orc, rows, cols, w_dtype, w0_dtype, sdq):
    if rows == 11008 and w_dtype != w0_dtype:
        pytest.skip("full size once per dtype")
    W = torch.from_numpy(_weights(rows + cols, rows, cols)).to(w_dtype)
    got = aw.awsrc_rtn_quantize(W.cuda(), sdq=sdq, w0_dtype=w0_dtype)
    torch.cuda.synchronize()
    want = orc.rtn_quantize(W.float().numpy(), sdq=sdq)
    assert np.array_equal(got["codes"].cpu().numpy(), _pack(want["q"]))
    assert np.array_equal(got["scales"].cpu().numpy().view(np.uint16), want["s16"])
    if sdq:
        assert np.array_equal(got["sdq_codes"].cpu().numpy(), want["c8"])
        assert np.array_equal(got["sdq_consts"].cpu().numpy().view(np.uint32), want["consts"].view(np.uint32))
    W0 = torch.from_numpy(want["W0"]).to(w0_dtype)
    assert torch.equal(got["W0"].cpu().view(torch.int16 if w0_dtype == torch.bfloat16 else torch.int32),
                       W0.view(torch.int16 if w0_dtype == torch.bfloat16 else torch.int32))


@pytest.mark.parametrize("sdq", [False, True])
def test_backbone_batch_matches_oracle(aw, orc, sdq):
    """Several modules in one call (two dtype runs, so two launches; shapes
    with a partial SDQ block and a zero group): every output equals the oracle's
    and the single call's bit for bit."""
    shapes = [(40, 512), (300, 1024), (7, 384), (256, 2048)]
    dts = [torch.bfloat16, torch.bfloat16, torch.float32, torch.float32]
    Ws = [torch.from_numpy(_weights(7 * i + r, r, c)).to(dt).cuda() for i, ((r, c), dt) in enumerate(zip(shapes, dts))]
    got = aw.awsrc_rtn_quantize_batch(Ws, sdq=sdq)
    torch.cuda.synchronize()
    for W, g in zip(Ws, got):
        single = aw.awsrc_rtn_quantize(W, sdq=sdq)
        for key in single:
            assert torch.equal(single[key].view(torch.uint8), g[key].view(torch.uint8)), key
        want = orc.rtn_quantize(W.float().cpu().numpy(), sdq=sdq)
        assert np.array_equal(g["codes"].cpu().numpy(), _pack(want["q"]))
        assert np.array_equal(g["scales"].cpu().numpy().view(np.uint16), want["s16"])
        if sdq:
            assert np.array_equal(g["sdq_codes"].cpu().numpy(), want["c8"])
            assert np.array_equal(g["sdq_consts"].cpu().numpy().view(np.uint32), want["consts"].view(np.uint32))
        W0 = torch.from_numpy(want["W0"]).to(W.dtype)
        itype = torch.int16 if W.dtype == torch.bfloat16 else torch.int32
        assert torch.equal(g["W0"].cpu().view(itype), W0.view(itype))


def test_backbone_batch_of_many_modules(aw):
    """More modules than one launch takes (20 > 16): the call splits into
    launches and every output still equals the single call's."""
    Ws = [torch.from_numpy(_weights(100 + i, 3 + i % 5, 128 * (1 + i % 3))).to(torch.bfloat16).cuda()
          for i in range(20)]
    for sdq in (False, True):
        got = aw.awsrc_rtn_quantize_batch(Ws, sdq=sdq)
        for W, g in zip(Ws, got):
            single = aw.awsrc_rtn_quantize(W, sdq=sdq)
            for key in single:
                assert torch.equal(single[key].view(torch.uint8), g[key].view(torch.uint8)), key


def test_sdq_savings_returned_to_the_sidecar_budget(aw, orc):
    """Sec. 3.3 end to end on one Qwen2.5-3B-shaped layer: the RTN-INT4 backbone
    with SDQ scales (W0 from the double-quantised scales), the encoder against
    that W0, and AWSRC-U selection at the rate that gives the metadata bytes SDQ
    saves to the records. Backbone metadata plus stream must fit the budget of
    binary16 scales plus a 0.162 bits/weight sidecar, the stream must hold more
    records than at 0.162 bits/weight, and the oracle must write the same stream."""
    from synth import WORKLOADS, make_layer
    wl = WORKLOADS["qwen2.5-3b_layer"]
    mods = make_layer(wl, layer=1, device="cuda")
    for m in mods:
        m["W0"] = aw.awsrc_rtn_quantize(m["W"], sdq=True)["W0"]
    shapes = [(m["rows"], m["cols"]) for m in mods]
    N = sum(r * c for r, c in shapes)
    kw = dict(C=wl.C, P=wl.P, b=wl.b, S=wl.S)
    prm, oprm = aw.params(**kw), orc.params(**kw)
    cands = aw.awsrc_encode_tiles(prm, mods)
    assert aw.awsrc_workspace_status(cands._awsrc_workspace) == 0
    rate2, saved = aw.awsrc_rate_with_sdq_savings(shapes, 0.162)
    meta_fp16 = sum(aw.awsrc_backbone_metadata_bytes(r, c, False) for r, c in shapes)
    meta_sdq = sum(aw.awsrc_backbone_metadata_bytes(r, c, True) for r, c in shapes)
    assert saved == meta_fp16 - meta_sdq > 0
    stream, counts, nbytes = aw.awsrc_select_records(prm, mods, cands, [rate2])
    _, counts0, _ = aw.awsrc_select_records(prm, mods, cands, [0.162])
    assert meta_sdq + int(nbytes[0]) <= meta_fp16 + orc.budget_bytes(0.162, N)
    assert int(counts.sum()) > int(counts0.sum())
    got = aw.candidates_to_numpy(cands)
    ostream, ocounts, _ = orc.select_records(oprm, shapes, got, [rate2])
    assert list(counts.cpu().numpy()) == list(ocounts)
    assert bytes(stream.cpu().numpy()[: int(nbytes[0])]) == ostream
