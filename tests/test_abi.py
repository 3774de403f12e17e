"""CPU checks of the C ABI library: it loads without a GPU, exports every entry
point declared in include/awsrc.h, and its host-only helpers (byte accounting,
argument validation) agree with the oracle. No compute call is made."""
import ctypes as ct
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "awsrc.h")


@pytest.fixture(scope="module")
def libpath():
    import __graft_entry__
    return __graft_entry__._cuda_build_module().build()


def declared_symbols():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(awsrc_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_three_steps():
    syms = declared_symbols()
    for s in ("awsrc_encode_tiles", "awsrc_select_records", "awsrc_decode_apply"):
        assert s in syms


def test_library_exports_every_declared_symbol(libpath):
    out = subprocess.run(["nm", "-D", "--defined-only", libpath], capture_output=True, text=True,
                         check=True).stdout
    exported = set(re.findall(r"\bT (awsrc_\w+)", out))
    missing = [s for s in declared_symbols() if s not in exported]
    assert not missing, f"declared but not exported: {missing}"
    lib = ct.CDLL(libpath)
    for s in declared_symbols():
        assert hasattr(lib, s)


def test_host_byte_accounting_matches_oracle(libpath, orc):
    import paper_2608_23144_gb300 as aw
    for C, P, b, S, b_e, smode in [(64, 4, 4, 256, 8, 0), (64, 4, 4, 256, 16, 1), (16, 4, 4, 16, 8, 0),
                                   (128, 2, 4, 2, 8, 0), (8, 8, 8, 65536, 3, 0)]:
        for T in (1, 2, 2048, 1_204_224, 152_174_592, 487_587_840):
            p = aw.params(C=C, P=P, b=b, S=S, b_e=b_e, scale_mode=smode)
            q = orc.params(C=C, P=P, b=b, S=S, b_e=b_e, scale_mode=smode)
            assert aw.awsrc_record_bytes(p, T) == orc.record_bytes(q, T)
    for n in (1, 7, 108, 252):
        assert aw.awsrc_header_bytes(n) == orc.header_bytes(n)


def test_host_validation_rejects_bad_arguments(libpath):
    import paper_2608_23144_gb300 as aw
    lib = aw.lib
    n = ct.c_size_t()
    mods = (aw.Module * 1)()
    mods[0].rows, mods[0].cols = 8, 96   # 96 is not a multiple of C = 64
    p = aw.params(C=64)
    assert lib.awsrc_encode_workspace_bytes(ct.byref(p), 1, mods, ct.byref(n)) == 2     # SHAPE
    mods[0].cols = 128
    assert lib.awsrc_encode_workspace_bytes(ct.byref(p), 1, mods, ct.byref(n)) == 0
    assert n.value > 0
    assert lib.awsrc_encode_workspace_bytes(ct.byref(aw.params(C=48)), 1, mods, ct.byref(n)) == 2
    assert lib.awsrc_encode_workspace_bytes(ct.byref(aw.params(P=9)), 1, mods, ct.byref(n)) == 3
    assert lib.awsrc_encode_workspace_bytes(ct.byref(aw.params(b=1)), 1, mods, ct.byref(n)) == 3
    assert lib.awsrc_encode_workspace_bytes(ct.byref(aw.params(S=70000)), 1, mods, ct.byref(n)) == 3
    assert lib.awsrc_encode_workspace_bytes(ct.byref(aw.params(scale_mode=1, b_e=8)), 1, mods, ct.byref(n)) == 3
    assert lib.awsrc_encode_workspace_bytes(ct.byref(aw.params(ridge_rel=-1.0)), 1, mods, ct.byref(n)) == 1
    assert lib.awsrc_encode_workspace_bytes(ct.byref(p), 0, mods, ct.byref(n)) == 1
    # encode with NULL tensors is refused before any launch
    assert lib.awsrc_encode_tiles(ct.byref(p), 1, mods, None, None, 0, None) == 1
    # a budget below the header: 8x128 weights at 0.01 bpw -> 1 byte < 48
    r = (ct.c_double * 1)(0.01)
    assert lib.awsrc_stream_capacity(ct.byref(p), 1, mods, r, 1, ct.byref(n)) == 4
    r = (ct.c_double * 1)(8.0)
    assert lib.awsrc_stream_capacity(ct.byref(p), 1, mods, r, 1, ct.byref(n)) == 0
    # U takes exactly one rate
    r2 = (ct.c_double * 2)(4.0, 8.0)
    assert lib.awsrc_stream_capacity(ct.byref(p), 1, mods, r2, 2, ct.byref(n)) == 3
    assert lib.awsrc_status_string(4) == b"byte budget smaller than the stream header"


def test_stream_capacity_matches_oracle_budget(libpath, orc):
    import paper_2608_23144_gb300 as aw
    lib = aw.lib
    shapes = [(2048, 2048), (256, 2048), (256, 2048), (2048, 2048), (11008, 2048), (11008, 2048), (2048, 11008)]
    mods = (aw.Module * len(shapes))()
    for i, (r, c) in enumerate(shapes):
        mods[i].rows, mods[i].cols = r, c
    p = aw.params(C=64, S=4096)
    q = orc.params(C=64, S=4096)
    n = ct.c_size_t()
    rates = (ct.c_double * 1)(0.162)
    assert lib.awsrc_stream_capacity(ct.byref(p), len(shapes), mods, rates, 1, ct.byref(n)) == 0
    N = sum(r * c for r, c in shapes)
    T = N // 64
    B = orc.budget_bytes(0.162, N)
    h, L = orc.header_bytes(len(shapes)), orc.record_bytes(q, T)
    quotas = [((B - h) * r * c) // N for r, c in shapes]
    assert n.value == h + sum(qm // L for qm in quotas) * L
    assert n.value <= B


def test_misaligned_pointers_are_refused_before_any_launch(libpath):
    """Pointer values are only compared here (no device memory exists): each
    call must return INVALID_ARG on the host, before touching the GPU."""
    import paper_2608_23144_gb300 as aw
    lib = aw.lib
    p = aw.params(C=64, S=64)
    mods = (aw.Module * 1)()
    mods[0].rows, mods[0].cols = 8, 128
    mods[0].w_dtype = mods[0].w0_dtype = aw.DTYPE_BF16
    mods[0].W, mods[0].W0, mods[0].act = 0x10000, 0x20000, 0x30000
    big = 1 << 40
    assert lib.awsrc_encode_tiles(ct.byref(p), 1, mods, 0x40000, 0x50001, big, None) == 1    # workspace
    assert lib.awsrc_encode_tiles(ct.byref(p), 1, mods, 0x40002, 0x50000, big, None) == 1    # candidates
    mods[0].W = 0x10001                                                                      # BF16 needs 2
    assert lib.awsrc_encode_tiles(ct.byref(p), 1, mods, 0x40000, 0x50000, big, None) == 1
    mods[0].W, mods[0].act = 0x10000, 0x30002                                                # f32 needs 4
    assert lib.awsrc_encode_tiles(ct.byref(p), 1, mods, 0x40000, 0x50000, big, None) == 1
    mods[0].act = 0x30000
    what = (ct.c_void_p * 1)(0x60008)                                                        # W_hat needs 16
    assert lib.awsrc_decode_apply(ct.byref(p), 1, mods, 0x70000, 1 << 20, 0, what, aw.DTYPE_BF16,
                                  aw.DECODE_DENSE, 0x80000, big, None) == 1
    what[0] = 0x60000
    mods[0].W0 = 0x20008                                                                     # dense W0 needs 16
    assert lib.awsrc_decode_apply(ct.byref(p), 1, mods, 0x70000, 1 << 20, 0, what, aw.DTYPE_BF16,
                                  aw.DECODE_DENSE, 0x80000, big, None) == 1
    mods[0].W0 = 0x20000
    assert lib.awsrc_decode_apply(ct.byref(p), 1, mods, 0x70000, 1 << 20, 0, what, aw.DTYPE_BF16,
                                  aw.DECODE_DENSE, 0x80040, big, None) == 1                  # workspace


def test_backbone_metadata_bytes(libpath):
    """Host-only byte count of the backbone's scale metadata (Sec. 3.3):
    binary16 per group of 128, or SDQ's byte per group plus 8 per 256 groups."""
    import paper_2608_23144_gb300 as aw
    G = 11008 * 2048 // 128
    assert aw.awsrc_backbone_metadata_bytes(11008, 2048, False) == 2 * G
    assert aw.awsrc_backbone_metadata_bytes(11008, 2048, True) == G + 8 * 688
    assert aw.awsrc_backbone_metadata_bytes(4, 100, True) == -1
    assert aw.awsrc_backbone_metadata_bytes(1, 128, True) == 1 + 8


@pytest.mark.parametrize("rate", [0.0, 0.05, 0.162, 0.25, 1.0])
def test_rate_with_sdq_savings_gives_the_saved_bytes_to_the_sidecar(libpath, orc, rate):
    """Sec. 3.3: the metadata bytes SDQ saves against binary16 scales go to the
    residual records under an unchanged total. The returned rate's budget
    (Eq. 5, floor(rate N / 8)) must be exactly the old budget plus the saving,
    counted here from the two metadata layouts (2 bytes per group of 128, or 1
    per group plus 8 per 256 groups)."""
    import math
    import paper_2608_23144_gb300 as aw
    from synth.workloads import _QWEN3B, _QWEN32B
    for shapes in ([(r, c) for _, r, c in _QWEN3B], [(r, c) for _, r, c in _QWEN32B], [(3, 128), (1, 384)]):
        N = sum(r * c for r, c in shapes)
        saved = 0
        for r, c in shapes:
            G = r * c // 128
            saved += 2 * G - (G + 8 * math.ceil(G / 256))
        if orc.budget_bytes(rate, N) + saved < 0:     # SDQ's block constants cost more than it saves
            with pytest.raises(aw.AwsrcError) as ei:
                aw.awsrc_rate_with_sdq_savings(shapes, rate)
            assert ei.value.status == 4
            continue
        r2, got_saved = aw.awsrc_rate_with_sdq_savings(shapes, rate)
        assert got_saved == saved
        assert orc.budget_bytes(r2, N) == orc.budget_bytes(rate, N) + saved
        assert (r2 >= rate) == (saved >= 0)
    with pytest.raises(aw.AwsrcError):
        aw.awsrc_rate_with_sdq_savings([(4, 100)], 0.1)       # cols not a multiple of 128
    with pytest.raises(aw.AwsrcError):
        aw.awsrc_rate_with_sdq_savings([(4, 128)], -1.0)


def test_serving_and_diagnostic_arguments_are_refused_on_the_host(libpath):
    """Pointer values are only compared (no device memory exists): the backbone
    quantiser, the packed GEMV and the reciprocal check return INVALID_ARG or
    SHAPE on the host, before any launch."""
    import paper_2608_23144_gb300 as aw
    lib = aw.lib
    bf16 = aw.DTYPE_BF16
    # awsrc_rtn_quantize: cols % 128, 16-byte W and W0, 4-byte codes
    assert lib.awsrc_rtn_quantize(8, 100, 0x10000, bf16, 0, 0x20000, 0x30000, None, None, 0x40000, bf16, None) == 2
    assert lib.awsrc_rtn_quantize(8, 128, 0x10008, bf16, 0, 0x20000, 0x30000, None, None, 0x40000, bf16, None) == 1
    assert lib.awsrc_rtn_quantize(8, 128, 0x10000, bf16, 0, 0x20002, 0x30000, None, None, 0x40000, bf16, None) == 1
    assert lib.awsrc_rtn_quantize(8, 128, 0x10000, bf16, 0, 0x20000, 0x30000, None, None, 0x40004, bf16, None) == 1
    assert lib.awsrc_rtn_quantize(8, 128, 0x10000, bf16, 2, 0x20000, 0x30000, None, None, 0x40000, bf16, None) == 1
    # awsrc_rtn_quantize_batch: every task is checked before anything runs
    from paper_2608_23144_gb300._binding import RtnTask
    ok = RtnTask(8, 128, 0x10000, bf16, 0, 0x20000, 0x30000, None, None, 0x40000, bf16, 0)
    bad = RtnTask(8, 100, 0x10000, bf16, 0, 0x20000, 0x30000, None, None, 0x40000, bf16, 0)
    assert lib.awsrc_rtn_quantize_batch(0, (RtnTask * 1)(ok), None) == 1
    assert lib.awsrc_rtn_quantize_batch(2, (RtnTask * 2)(ok, bad), None) == 2
    ok2 = RtnTask(8, 128, 0x10000, bf16, 0, 0x20002, 0x30000, None, None, 0x40000, bf16, 0)
    assert lib.awsrc_rtn_quantize_batch(2, (RtnTask * 2)(ok, ok2), None) == 1
    # awsrc_packed_gemv: M in [1, 8], module index, 16-byte x, 4-byte codes
    from paper_2608_23144_gb300._binding import PackedWeights, shape_modules
    p = aw.params(C=64, S=64)
    mods = shape_modules([(8, 128)])
    pw = PackedWeights(0x10000, 0x20000, None, None, 0, 0)
    assert lib.awsrc_packed_gemv(ct.byref(p), 1, mods, 0, ct.byref(pw), None, 0, 9, 0x30000, 0x40000, None) == 1
    assert lib.awsrc_packed_gemv(ct.byref(p), 1, mods, 1, ct.byref(pw), None, 0, 1, 0x30000, 0x40000, None) == 1
    assert lib.awsrc_packed_gemv(ct.byref(p), 1, mods, 0, ct.byref(pw), None, 0, 1, 0x30008, 0x40000, None) == 1
    pw.codes = 0x10002
    assert lib.awsrc_packed_gemv(ct.byref(p), 1, mods, 0, ct.byref(pw), None, 0, 1, 0x30000, 0x40000, None) == 1
    # awsrc_packed_gemv_batch: 1 <= n_task <= 16 (more: UNSUPPORTED), each task checked like a single call
    from paper_2608_23144_gb300._binding import GemvTask
    pw.codes = 0x10000
    tasks = (GemvTask * 17)(*[GemvTask(0, 0, pw, 0x30000, 0x40000 + 0x100 * i) for i in range(17)])
    assert lib.awsrc_packed_gemv_batch(ct.byref(p), 1, mods, 0, tasks, None, 0, 1, None) == 1
    assert lib.awsrc_packed_gemv_batch(ct.byref(p), 1, mods, 17, tasks, None, 0, 1, None) == 3
    assert lib.awsrc_packed_gemv_batch(ct.byref(p), 1, mods, 2, None, None, 0, 1, None) == 1
    assert lib.awsrc_packed_gemv_batch(ct.byref(p), 1, mods, 2, tasks, None, 0, 0, None) == 1
    tasks[1].m = 1
    assert lib.awsrc_packed_gemv_batch(ct.byref(p), 1, mods, 2, tasks, None, 0, 1, None) == 1
    tasks[1].m, tasks[1].x = 0, 0x30004
    assert lib.awsrc_packed_gemv_batch(ct.byref(p), 1, mods, 2, tasks, None, 0, 1, None) == 1
    # awsrc_verify_reciprocal: null, misaligned counter, empty-range order
    assert lib.awsrc_verify_reciprocal(0, 1, None, None) == 1
    assert lib.awsrc_verify_reciprocal(0, 1, 0x50004, None) == 1
    assert lib.awsrc_verify_reciprocal(2, 1, 0x50000, None) == 1


def test_size_limits_are_refused_before_any_product_overflows(libpath):
    """Tile indices are 32-bit and one RTN launch covers at most 2^46 weights:
    shapes past either limit return UNSUPPORTED (or -1) on the host, including
    shapes whose rows * cols would overflow int64."""
    import paper_2608_23144_gb300 as aw
    from paper_2608_23144_gb300._binding import shape_modules
    lib = aw.lib
    p = aw.params(C=64, S=64)
    n = ct.c_size_t()
    ws = lambda shapes: lib.awsrc_encode_workspace_bytes(ct.byref(p), len(shapes), shape_modules(shapes),
                                                         ct.byref(n))
    assert ws([((1 << 32) - 1, 64)]) == 0                  # 2^32 - 1 tiles: the largest call
    assert ws([(1 << 32, 64)]) == 3                        # 2^32 tiles
    assert ws([((1 << 31), 64), ((1 << 31), 64)]) == 3     # the limit is over the whole call
    assert ws([(1 << 40, 1 << 40)]) == 3                   # rows * cols / C overflows int64
    assert lib.awsrc_backbone_metadata_bytes(1 << 18, 1 << 28, 0) == 2 * (1 << 39)
    assert lib.awsrc_backbone_metadata_bytes(1 << 19, 1 << 28, 0) == -1
    assert lib.awsrc_backbone_metadata_bytes(1 << 40, 1 << 40, 1) == -1
    bf16 = aw.DTYPE_BF16
    assert lib.awsrc_rtn_quantize(1 << 40, 1 << 40, 0x10000, bf16, 0, 0x20000, 0x30000, None, None, 0x40000,
                                  bf16, None) == 3
    # the decoder that allocates nothing applies the same 32-bit tile limit
    outs = (ct.c_void_p * 2)(0x20000, 0x30000)
    nd = lambda shapes: lib.awsrc_decode_apply_inplace_noalloc(ct.byref(p), len(shapes), shape_modules(shapes),
                                                               0x10000, 1 << 20, 0, outs, None)
    assert nd([(1 << 32, 64)]) == 3
    assert nd([(1 << 31, 64), (1 << 31, 64)]) == 3
    assert nd([(1 << 40, 1 << 40)]) == 3
