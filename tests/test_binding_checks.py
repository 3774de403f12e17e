"""The Python binding refuses, on the host and before any pointer crosses the
C ABI, tensors whose shape, element type, size or device disagree with the
module shapes the kernels index them by (a mismatch would otherwise be read
or written out of bounds on the device). CPU and meta tensors stand in for
device memory: every call here must stop at one of these checks."""
import pytest
import torch

import paper_2608_23144_gb300 as aw

ROWS, COLS = 8, 128


def module(**over):
    m = {"W": torch.zeros(ROWS, COLS, dtype=torch.bfloat16), "W0": torch.zeros(ROWS, COLS, dtype=torch.bfloat16),
         "act": torch.ones(COLS, dtype=torch.float32), "fisher": None}
    m.update(over)
    return m


PRM = aw.params(C=64, P=4, b=4, S=64)
T = ROWS * COLS // 64


@pytest.mark.parametrize("over,exc,msg", [
    (dict(W=torch.zeros(COLS, ROWS, dtype=torch.bfloat16)), ValueError, r"\['W'\] has shape"),
    (dict(act=torch.ones(COLS, dtype=torch.float64)), TypeError, r"\['act'\] must be torch.float32"),
    (dict(act=torch.ones(COLS - 1, dtype=torch.float32)), ValueError, r"\['act'\] holds 127"),
    (dict(fisher=torch.ones(ROWS, COLS - 64)), ValueError, r"\['fisher'\] has shape"),
    (dict(fisher=torch.ones(ROWS, COLS, dtype=torch.float16)), TypeError, r"\['fisher'\] must be"),
    (dict(act=torch.ones(COLS, dtype=torch.float32, device="meta")), ValueError, r"\['act'\] is on meta"),
    (dict(W0=torch.zeros(ROWS * COLS, dtype=torch.bfloat16)), ValueError, r"must be 2-D"),
])
def test_encoder_modules_are_checked(over, exc, msg):
    with pytest.raises(exc, match=msg):
        aw.awsrc_encode_tiles(PRM, [module(**over)])


def test_encoder_output_is_checked():
    with pytest.raises(ValueError, match=r"out holds 160 elements, at least 256"):
        aw.awsrc_encode_tiles(PRM, [module()], out=torch.empty(10, 16, dtype=torch.uint8))
    with pytest.raises(TypeError, match=r"out must be torch.uint8"):
        aw.awsrc_encode_tiles(PRM, [module()], out=torch.empty(T, 4, dtype=torch.int32))


def test_selection_buffers_are_checked():
    mods = [module()]
    with pytest.raises(ValueError, match=r"cands holds"):
        aw.awsrc_select_records(PRM, mods, torch.empty(T - 1, 16, dtype=torch.uint8), [0.5])
    with pytest.raises(TypeError, match=r"cands must be torch.uint8"):
        aw.awsrc_select_records(PRM, mods, torch.empty(T, 4, dtype=torch.float32), [0.5])
    cands = torch.empty(T, 16, dtype=torch.uint8)
    with pytest.raises(TypeError, match=r"counts must be torch.int64"):
        aw.awsrc_select_records(PRM, mods, cands, [0.5], counts=torch.empty(1, dtype=torch.int32))
    with pytest.raises(TypeError, match=r"nbytes must be torch.int64"):
        aw.awsrc_select_records(PRM, mods, cands, [0.5], nbytes=torch.empty(1, dtype=torch.float64))
    with pytest.raises(TypeError, match=r"out must be torch.uint8"):
        aw.awsrc_select_records(PRM, mods, cands, [0.5], out=torch.empty(64, dtype=torch.int16))


def test_decoder_outputs_are_checked():
    mods = [module(), module(W0=torch.zeros(4, 64, dtype=torch.bfloat16))]
    stream = torch.zeros(256, dtype=torch.uint8)
    good = [torch.empty(ROWS, COLS, dtype=torch.bfloat16), torch.empty(4, 64, dtype=torch.bfloat16)]
    with pytest.raises(ValueError, match=r"1 outputs for 2 modules"):
        aw.awsrc_decode_apply(PRM, mods, stream, 0, outs=good[:1])
    with pytest.raises(ValueError, match=r"outs\[1\] has shape \(4, 32\)"):
        aw.awsrc_decode_apply(PRM, mods, stream, 0, outs=[good[0], torch.empty(4, 32, dtype=torch.bfloat16)])
    with pytest.raises(TypeError, match=r"outs\[1\] must be torch.bfloat16"):
        aw.awsrc_decode_apply(PRM, mods, stream, 0, outs=[good[0], torch.empty(4, 64)])
    with pytest.raises(TypeError, match=r"out_dtype must be"):
        aw.awsrc_decode_apply(PRM, mods, stream, 0, out_dtype=torch.float16)
    with pytest.raises(ValueError, match=r"1 outputs for 2 modules"):
        aw.awsrc_decode_apply_inplace_noalloc(PRM, mods, stream, 0, good[:1])
    with pytest.raises(TypeError, match=r"outs\[0\] must be torch.bfloat16"):
        aw.awsrc_decode_apply_inplace_noalloc(PRM, mods, stream, 0, [torch.empty(ROWS, COLS), good[1]])


def test_backbone_and_gemv_buffers_are_checked():
    with pytest.raises(ValueError, match=r"W must be 2-D"):
        aw.awsrc_rtn_quantize(torch.zeros(ROWS * COLS))
    G = ROWS * COLS // 128
    bb = {"codes": torch.empty(ROWS * COLS // 2, dtype=torch.uint8), "scales": torch.empty(G, dtype=torch.int16),
          "W0": torch.empty(ROWS, COLS)}
    with pytest.raises(ValueError, match=r"out\['codes'\] holds"):
        aw.awsrc_rtn_quantize(torch.zeros(ROWS, COLS), out={**bb, "codes": bb["codes"][:-1]})
    with pytest.raises(TypeError, match=r"out\['sdq_codes'\] must be torch.int8"):
        aw.awsrc_rtn_quantize(torch.zeros(ROWS, COLS), sdq=True,
                              out={**bb, "sdq_codes": torch.empty(G, dtype=torch.uint8),
                                   "sdq_consts": torch.empty(2, dtype=torch.float32)})
    shapes = [(ROWS, COLS)]
    x = torch.zeros(1, COLS)
    with pytest.raises(TypeError, match=r"x must be torch.float32"):
        aw.awsrc_packed_gemv(PRM, shapes, 0, bb, x.double())
    with pytest.raises(ValueError, match=r"not a whole number of rows"):
        aw.awsrc_packed_gemv(PRM, shapes, 0, bb, torch.zeros(COLS + 1))
    with pytest.raises(ValueError, match=r"y has shape"):
        aw.awsrc_packed_gemv(PRM, shapes, 0, bb, x, y=torch.empty(1, ROWS - 1))
    with pytest.raises(ValueError, match=r"backbone\['codes'\] holds"):
        aw.awsrc_packed_gemv(PRM, shapes, 0, {**bb, "codes": bb["codes"][:8]}, x)
    with pytest.raises(TypeError, match=r"backbone\['scales'\] must be torch.int16"):
        aw.awsrc_packed_gemv(PRM, shapes, 0, {**bb, "scales": bb["scales"].float()}, x)
    with pytest.raises(TypeError, match=r"sidecar must be torch.uint8"):
        aw.awsrc_packed_gemv(PRM, shapes, 0, bb, x, sidecar=torch.empty(8, dtype=torch.int32))
