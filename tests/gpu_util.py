"""Helpers shared by the GPU parity tests: build seeded inputs once, run the CUDA
path through the C ABI binding and the oracle on the same arrays, compare."""
import numpy as np
import torch


def to_dev(mods, dev="cuda"):
    return [{k: (v.to(dev) if torch.is_tensor(v) else v) for k, v in m.items()} for m in mods]


def host_f32(t):
    return None if t is None else t.detach().float().cpu().numpy()


def params_pair(aw, orc, **kw):
    return aw.params(**kw), orc.params(**kw)


def oracle_encode(orc, oprm, mods, masks=None, tiles_per_module=None):
    if masks is None:
        masks = orc.basis_masks(oprm)
    out = []
    for i, m in enumerate(mods):
        tl = None if tiles_per_module is None else tiles_per_module[i]
        out.append(orc.encode_tiles(oprm, host_f32(m["W"]), host_f32(m["W0"]), host_f32(m["act"]),
                                    fisher=host_f32(m.get("fisher")), w_act=m.get("w_act", 1.0),
                                    w_fisher=m.get("w_fisher", 0.0), tiles=tl, masks=masks))
    return out


def assert_candidates_equal(got, want, label=""):
    """Bit-exact equality of every field (gain compared by its bit pattern)."""
    assert got.shape == want.shape, label
    bad = np.nonzero((got["gain"].view(np.uint32) != want["gain"].view(np.uint32)) |
                     (got["seed"] != want["seed"]) | (got["scale"] != want["scale"]) |
                     np.any(got["code"] != want["code"], axis=1))[0]
    if len(bad):
        i = bad[0]
        raise AssertionError(f"{label}: {len(bad)} of {len(got)} tiles differ; first tile {i}: "
                             f"gpu {got[i]} oracle {want[i]}")


def block_tiles(rng, rows, n_cb, block_rows=128):
    """Tile indices of one whole block of the C = 64 search (block_rows
    consecutive rows of one column block, chosen at random), plus every tile of
    the module's first row."""
    nb = (rows + block_rows - 1) // block_rows
    rb, cb = int(rng.integers(nb)), int(rng.integers(n_cb))
    r = np.arange(rb * block_rows, min(rows, (rb + 1) * block_rows))
    return np.concatenate([r * n_cb + cb, np.arange(n_cb)])
