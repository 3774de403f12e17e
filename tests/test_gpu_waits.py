"""The search kernels' bounded waits, made to run out on purpose.

Every wait inside the tcgen05 search (for a chunk's bulk copies, for its
tensor-core results, for the release of shared buffers) gives up after a time
limit; the block then records the timeout bit of the workspace's fault word,
waits for its own copies and tensor-core work still in flight, frees its
tensor memory and exits, so that the GPU context stays usable. Here the limit
is shortened to 200 us and the producer issues no copies from one seed chunk
on, so nothing ever completes that chunk: the waits for it must run out, the
call must report bit 2, and the next normal call on the same GPU must give
the same candidates as before, which match the oracle's."""
import numpy as np
import pytest
import torch

from gpu_util import assert_candidates_equal, host_f32

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def aw():
    import paper_2608_23144_gb300 as aw
    assert torch.cuda.is_available()
    return aw


@pytest.mark.parametrize("shape,stall", [((4096, 512), 5), ((128, 64), 0), ((1000, 256), 3)])
def test_bounded_wait_runs_out_and_is_reported(aw, orc, shape, stall):
    from synth import make_module
    m = make_module(*shape, seed=31, device="cuda")
    prm = aw.params(C=64, P=4, b=4, S=4096)
    before = aw.awsrc_encode_tiles(prm, [m])
    ws = before._awsrc_workspace
    assert aw.awsrc_workspace_status(ws) == 0
    before = before.clone()
    aw.awsrc_set_wait_test(200_000, stall)
    try:
        aw.awsrc_encode_tiles(prm, [m], workspace=ws)
        flags = aw.awsrc_workspace_status(ws)
    finally:
        aw.awsrc_set_wait_test()
    assert flags & 4, f"the timeout was not reported (flags {flags:#x})"
    after = aw.awsrc_encode_tiles(prm, [m], workspace=ws)
    assert aw.awsrc_workspace_status(ws) == 0
    assert torch.equal(after, before)
    # and the candidates are the oracle's (the first and last rows)
    oprm = orc.params(C=64, P=4, b=4, S=4096)
    n_cb = shape[1] // 64
    T = shape[0] * n_cb
    tiles = np.unique(np.concatenate([np.arange(min(T, 2 * n_cb)), np.arange(T - n_cb, T)]))
    want = orc.encode_tiles(oprm, host_f32(m["W"]), host_f32(m["W0"]), host_f32(m["act"]), tiles=tiles,
                            masks=orc.basis_masks(oprm))
    assert_candidates_equal(aw.candidates_to_numpy(after)[tiles], want, f"after a timeout {shape}")
