"""Parity at the sizes of the larger workloads, sampled where the oracle cannot
run whole, in the launch configurations a user of those workloads runs:

* one Qwen2.5-32B-shaped layer (7 modules, 487,587,840 BF16 weights,
  7,618,560 tiles, S = 4096): AWSRC-U at 0.162 bits/weight — sampled tiles of
  every module re-searched by the oracle, the stream re-selected by the oracle
  byte for byte, every repaired weight decoded by the oracle;
* one Qwen2.5-7B-shaped layer and one Qwen2.5-32B-shaped layer with AWSRC-P_F
  (0.5/0.5 blend of normalised activation moments and Fisher diagonal):
  sampled tiles, the progressive stream at 0.05 / 0.10 / 0.162 / 0.25
  bits/weight re-selected by the oracle, and the smallest and largest
  prefixes decoded;
* three layers of the Qwen2.5-3B stack encoded layer by layer, then selected
  and decoded as one model of 21 modules (more than one launch group)."""
import numpy as np
import pytest
import torch

from gpu_util import assert_candidates_equal, block_tiles, host_f32

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


@pytest.fixture(scope="module")
def aw():
    import paper_2608_23144_gb300 as aw
    return aw


def _sample_tiles(rng, rows, n_cb, k=12):
    """Corner tiles, k random tiles, one whole 128-row block of the search
    kernel and the module's first row."""
    T_m = rows * n_cb
    return np.unique(np.concatenate([[0, n_cb - 1, T_m - n_cb, T_m - 1], rng.choice(T_m, k, replace=False),
                                     block_tiles(rng, rows, n_cb)]))


def _check_sampled(orc, oprm, got, mods, C, seed):
    masks = orc.basis_masks(oprm)
    rng = np.random.default_rng(seed)
    off = 0
    for m in mods:
        T_m = m["rows"] * m["cols"] // C
        tiles = _sample_tiles(rng, m["rows"], m["cols"] // C)
        want = orc.encode_tiles(oprm, host_f32(m["W"]), host_f32(m["W0"]), host_f32(m["act"]),
                                fisher=host_f32(m.get("fisher")), w_act=m.get("w_act", 1.0),
                                w_fisher=m.get("w_fisher", 0.0), tiles=tiles, masks=masks)
        assert_candidates_equal(got[off + tiles], want, m["name"])
        off += T_m
    assert off == len(got)


def test_qwen32b_layer_u(aw, orc):
    from synth import WORKLOADS, make_layer
    wl = WORKLOADS["qwen2.5-32b_stack"]
    mods = make_layer(wl, layer=5, device="cuda")
    prm, oprm = aw.params(C=wl.C, P=wl.P, b=wl.b, S=wl.S), orc.params(C=wl.C, P=wl.P, b=wl.b, S=wl.S)
    cands = aw.awsrc_encode_tiles(prm, mods)
    assert aw.awsrc_workspace_status(cands._awsrc_workspace) == 0
    got = aw.candidates_to_numpy(cands)
    assert len(got) == wl.tiles_per_layer == 7_618_560
    _check_sampled(orc, oprm, got, mods, wl.C, seed=1)
    shapes = [(m["rows"], m["cols"]) for m in mods]
    stream, counts, nbytes = aw.awsrc_select_records(prm, mods, cands, [0.162])
    ostream, ocounts, _ = orc.select_records(oprm, shapes, got, [0.162])
    assert list(counts.cpu().numpy()) == list(ocounts)
    assert bytes(stream.cpu().numpy()[: int(nbytes[0])]) == ostream
    K = int(counts.sum())
    outs = aw.awsrc_decode_apply(prm, mods, stream, K)
    torch.cuda.synchronize()
    assert aw.awsrc_workspace_status(outs[0]._awsrc_workspace) == 0
    oouts, bad = orc.decode_apply(oprm, [host_f32(m["W0"]) for m in mods], ostream, K, out_bf16=True)
    assert bad == 0
    for g, o, m in zip(outs, oouts, mods):
        assert np.array_equal(g.float().cpu().numpy(), o), m["name"]


def test_qwen7b_layer_pf_prefixes(aw, orc):
    from synth import WORKLOADS, make_layer
    wl = WORKLOADS["qwen2.5-7b_stack_pf"]
    mods = make_layer(wl, layer=3, device="cuda")
    kw = dict(C=wl.C, P=wl.P, b=wl.b, S=wl.S, variant=1)
    prm, oprm = aw.params(**kw), orc.params(**kw)
    cands = aw.awsrc_encode_tiles(prm, mods)
    assert aw.awsrc_workspace_status(cands._awsrc_workspace) == 0
    got = aw.candidates_to_numpy(cands)
    assert len(got) == wl.tiles_per_layer
    _check_sampled(orc, oprm, got, mods, wl.C, seed=2)
    shapes = [(m["rows"], m["cols"]) for m in mods]
    rates = list(wl.rates)
    stream, counts, nbytes = aw.awsrc_select_records(prm, mods, cands, rates)
    ostream, ocounts, obytes = orc.select_records(oprm, shapes, got, rates)
    assert list(counts.cpu().numpy()) == list(ocounts)
    assert list(nbytes.cpu().numpy()) == list(obytes)
    assert bytes(stream.cpu().numpy()[: int(nbytes.max())]) == ostream
    W0s = [host_f32(m["W0"]) for m in mods]
    for K in (int(ocounts[0]), int(ocounts[-1])):   # the smallest and the largest prefix
        outs = aw.awsrc_decode_apply(prm, mods, stream, K)
        torch.cuda.synchronize()
        oouts, bad = orc.decode_apply(oprm, W0s, ostream, K, out_bf16=True)
        assert bad == 0
        for g, o, m in zip(outs, oouts, mods):
            assert np.array_equal(g.float().cpu().numpy(), o), (K, m["name"])


def test_qwen32b_layer_pf_prefixes(aw, orc):
    """The Qwen2.5-32B-shaped layer under AWSRC-P_F (the 0.5/0.5 blend of
    normalised activation moments and Fisher diagonal): sampled tiles, the
    progressive stream at 0.05 / 0.10 / 0.162 / 0.25 bits/weight re-selected by
    the oracle byte for byte, and the smallest and largest prefixes decoded."""
    from synth import WORKLOADS, make_layer
    from synth.workloads import make_module, module_seed
    wl = WORKLOADS["qwen2.5-32b_stack"]
    layer = 9
    mods = []
    for mi, (name, rows, cols) in enumerate(wl.shapes):
        m = make_module(rows, cols, seed=module_seed(wl.seed, layer, mi), device="cuda", w_dtype=wl.w_dtype,
                        outlier=wl.outlier, fisher=True, blend=(0.5, 0.5))
        m["name"] = name
        mods.append(m)
    kw = dict(C=wl.C, P=wl.P, b=wl.b, S=wl.S, variant=1)
    prm, oprm = aw.params(**kw), orc.params(**kw)
    cands = aw.awsrc_encode_tiles(prm, mods)
    assert aw.awsrc_workspace_status(cands._awsrc_workspace) == 0
    got = aw.candidates_to_numpy(cands)
    assert len(got) == wl.tiles_per_layer == 7_618_560
    _check_sampled(orc, oprm, got, mods, wl.C, seed=5)
    for m in mods:            # the decoder reads W0 only
        m["fisher"] = None
    shapes = [(m["rows"], m["cols"]) for m in mods]
    rates = [0.05, 0.10, 0.162, 0.25]
    stream, counts, nbytes = aw.awsrc_select_records(prm, mods, cands, rates)
    ostream, ocounts, obytes = orc.select_records(oprm, shapes, got, rates)
    assert list(counts.cpu().numpy()) == list(ocounts)
    assert list(nbytes.cpu().numpy()) == list(obytes)
    assert bytes(stream.cpu().numpy()[: int(nbytes.max())]) == ostream
    W0s = [host_f32(m["W0"]) for m in mods]
    for K in (int(ocounts[0]), int(ocounts[-1])):
        outs = aw.awsrc_decode_apply(prm, mods, stream, K)
        torch.cuda.synchronize()
        assert aw.awsrc_workspace_status(outs[0]._awsrc_workspace) == 0
        oouts, bad = orc.decode_apply(oprm, W0s, ostream, K, out_bf16=True)
        assert bad == 0
        for g, o, m in zip(outs, oouts, mods):
            assert np.array_equal(g.float().cpu().numpy(), o), (K, m["name"])
        del outs, oouts


def test_qwen3b_three_layers_as_one_model(aw, orc):
    from synth import WORKLOADS, make_layer
    wl = WORKLOADS["qwen2.5-3b_stack"]
    prm, oprm = aw.params(C=wl.C, P=wl.P, b=wl.b, S=wl.S), orc.params(C=wl.C, P=wl.P, b=wl.b, S=wl.S)
    mods, parts = [], []
    for layer in (0, 17, 35):          # encode layer by layer
        lm = make_layer(wl, layer=layer, device="cuda")
        c = aw.awsrc_encode_tiles(prm, lm)
        assert aw.awsrc_workspace_status(c._awsrc_workspace) == 0
        parts.append(aw.candidates_to_numpy(c))
        if layer == 17:
            _check_sampled(orc, oprm, parts[-1], lm, wl.C, seed=3)
        mods += lm
    got = np.concatenate(parts)
    cands = torch.from_numpy(got.view(np.uint8).reshape(-1, 16).copy()).cuda()
    shapes = [(m["rows"], m["cols"]) for m in mods]
    stream, counts, nbytes = aw.awsrc_select_records(prm, mods, cands, [0.162])
    ostream, ocounts, _ = orc.select_records(oprm, shapes, got, [0.162])
    assert list(counts.cpu().numpy()) == list(ocounts)
    assert bytes(stream.cpu().numpy()[: int(nbytes[0])]) == ostream
    K = int(counts.sum())
    outs = aw.awsrc_decode_apply(prm, mods, stream, K)
    torch.cuda.synchronize()
    oouts, bad = orc.decode_apply(oprm, [host_f32(m["W0"]) for m in mods], ostream, K, out_bf16=True)
    assert bad == 0
    for g, o, m in zip(outs, oouts, mods):
        assert np.array_equal(g.float().cpu().numpy(), o), m["name"]
