"""Full-size parity on one Qwen2.5-3B-shaped layer (7 modules, 77,070,336 BF16
weights, 1,204,224 tiles, S = 4096 seeds, AWSRC-U at 0.162 bits/weight) in the
launch configuration the benchmark times:

* encode: sampled tiles of every module re-searched by the oracle over all
  4096 seeds, every field bit for bit (one whole 128-row block of the search
  kernel, the module's first row, its corner tiles and random tiles);
* select: the oracle re-selects from the GPU's candidates; stream identical;
* decode: the oracle decodes the GPU's stream; every weight identical."""
import numpy as np
import pytest
import torch

from gpu_util import assert_candidates_equal, block_tiles, host_f32

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


@pytest.fixture(scope="module")
def layer():
    import paper_2608_23144_gb300 as aw
    from synth import WORKLOADS, make_layer
    wl = WORKLOADS["qwen2.5-3b_layer"]
    mods = make_layer(wl, layer=0, device="cuda")
    prm = aw.params(C=wl.C, P=wl.P, b=wl.b, S=wl.S)
    cands = aw.awsrc_encode_tiles(prm, mods)
    flags = aw.awsrc_workspace_status(cands._awsrc_workspace)
    return aw, wl, mods, prm, cands, flags


def test_fullsize_encode_sampled_tiles(layer, orc):
    aw, wl, mods, prm, cands, flags = layer
    assert flags == 0
    got = aw.candidates_to_numpy(cands)
    oprm = orc.params(C=wl.C, P=wl.P, b=wl.b, S=wl.S)
    masks = orc.basis_masks(oprm)
    rng = np.random.default_rng(0)
    off = 0
    for m in mods:
        T_m = m["rows"] * m["cols"] // wl.C
        n_cb = m["cols"] // wl.C
        tiles = np.unique(np.concatenate([[0, n_cb - 1, T_m - n_cb, T_m - 1],
                                          rng.choice(T_m, 20, replace=False),
                                          block_tiles(rng, m["rows"], n_cb)]))
        want = orc.encode_tiles(oprm, host_f32(m["W"]), host_f32(m["W0"]), host_f32(m["act"]),
                                tiles=tiles, masks=masks)
        assert_candidates_equal(got[off + tiles], want, m["name"])
        off += T_m
    assert off == len(got) == wl.tiles_per_layer
    # the search finds a positive-gain candidate for nearly every tile
    assert (got["gain"] > 0).mean() > 0.99


def test_fullsize_select_and_decode(layer, orc):
    aw, wl, mods, prm, cands, flags = layer
    oprm = orc.params(C=wl.C, P=wl.P, b=wl.b, S=wl.S)
    shapes = [(m["rows"], m["cols"]) for m in mods]
    stream, counts, nbytes = aw.awsrc_select_records(prm, mods, cands, [0.162])
    got = aw.candidates_to_numpy(cands)
    ostream, ocounts, obytes = orc.select_records(oprm, shapes, got, [0.162])
    assert list(counts.cpu().numpy()) == list(ocounts)
    gstream = bytes(stream.cpu().numpy()[: int(nbytes[0])])
    assert gstream == ostream
    N = wl.weights_per_layer
    assert len(gstream) <= orc.budget_bytes(0.162, N)
    K = int(counts.sum())
    outs = aw.awsrc_decode_apply(prm, mods, stream, K)
    torch.cuda.synchronize()
    oouts, bad = orc.decode_apply(oprm, [host_f32(m["W0"]) for m in mods], ostream, K, out_bf16=True)
    assert bad == 0
    for g, o, m in zip(outs, oouts, mods):
        assert np.array_equal(g.float().cpu().numpy(), o), m["name"]
    # the repaired layer is closer to W under the activation weights
    for g, m in zip(outs, mods):
        d = m["act"].double()[None, :]
        e0 = ((m["W"].double() - m["W0"].double()) ** 2 * d).sum().item()
        e1 = ((m["W"].double() - g.double()) ** 2 * d).sum().item()
        assert e1 < e0, m["name"]
