"""The library's own correctly rounded reciprocal (used for every D_k^-1 of the
LDL^T factorisations, Eq. 3) against CUDA's __frcp_rn, bit for bit, on every
binary32 pattern of its fast-path range [2^-125, 2^125) and on samples of the
inputs that take the fallback (zeros, subnormals, large values, negatives,
infinities and NaNs)."""
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def aw():
    import paper_2608_23144_gb300 as aw
    assert torch.cuda.is_available()
    return aw


def test_reciprocal_fast_path_is_exact_on_its_whole_range(aw):
    assert aw.awsrc_verify_reciprocal(0x01000000, 0x7D000000) == 0


@pytest.mark.parametrize("lo,hi", [(0x00000000, 0x01000000), (0x7D000000, 0x80000000),
                                   (0x80000000, 0x80100000), (0xFF7FF000, 0xFFFFFFFF)])
def test_reciprocal_fallback_ranges(aw, lo, hi):
    assert aw.awsrc_verify_reciprocal(lo, hi) == 0
