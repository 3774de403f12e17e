"""The decoder entry point that allocates nothing (awsrc_decode_apply_inplace_noalloc).

It exists for callers that may not allocate device memory — a model loader
whose engine has given all device memory to its own pool, a plain C program,
a recovery path — and keeps its scratch in a static device array of the
library. These tests call it through the C ABI twice in a row with different
streams and parameters (the array keeps the previous call's contents) and
compare every weight with the regular awsrc_decode_apply. This file is
collected last on purpose; it must pass on its own and after the others."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


def _case(aw, shapes, seed, w_dtype="bf16", rates=(1.0,), **kw):
    from synth import make_module
    pf = kw.get("variant", 0) == 1
    mods = [make_module(r, c, seed=seed + 11 * i, device="cuda", w_dtype=w_dtype, fisher=pf, blend=(0.5, 0.5))
            for i, (r, c) in enumerate(shapes)]
    prm = aw.params(**kw)
    cands = aw.awsrc_encode_tiles(prm, mods)
    stream, counts, nbytes = aw.awsrc_select_records(prm, mods, cands, list(rates))
    K = int(counts.sum()) if not pf else int(counts.max())
    return mods, prm, stream[: int(nbytes.max())].clone(), K


def test_noalloc_decode_matches_regular_decode_twice():
    import paper_2608_23144_gb300 as aw
    cases = [
        _case(aw, [(100, 256), (64, 128)], 1, C=64, P=4, b=4, S=64),
        _case(aw, [(40, 512), (96, 64), (7, 128)], 2, C=64, P=4, b=4, S=4096, gen_seed=99),
    ]
    for mods, prm, stream, K in cases:          # two calls in a row, different tables
        ref = aw.awsrc_decode_apply(prm, mods, stream, K, mode=aw.DECODE_DENSE)
        outs = [m["W0"].clone() for m in mods]
        aw.awsrc_decode_apply_inplace_noalloc(prm, mods, stream, K, outs)
        torch.cuda.synchronize()
        for a, b in zip(ref, outs):
            assert torch.equal(a, b)
        assert any(not torch.equal(o, m["W0"]) for o, m in zip(outs, mods))
    # a prefix of the first stream after the second call: stale table contents must not leak
    mods, prm, stream, K = cases[0]
    ref = aw.awsrc_decode_apply(prm, mods, stream, K // 2, mode=aw.DECODE_DENSE)
    outs = [m["W0"].clone() for m in mods]
    aw.awsrc_decode_apply_inplace_noalloc(prm, mods, stream, K // 2, outs)
    torch.cuda.synchronize()
    for a, b in zip(ref, outs):
        assert torch.equal(a, b)


def test_noalloc_decode_rejects_tables_beyond_its_limit():
    import paper_2608_23144_gb300 as aw
    mods = [{"W0": torch.zeros(4, 256, dtype=torch.bfloat16, device="cuda")}]
    prm = aw.params(C=256, P=8, S=8192)          # 8192 * 8 * 4 words > 131072
    stream = torch.zeros(64, dtype=torch.uint8, device="cuda")
    with pytest.raises(aw.AwsrcError) as ei:
        aw.awsrc_decode_apply_inplace_noalloc(prm, mods, stream, 0, [mods[0]["W0"]])
    assert ei.value.status == 3
    assert b"131072" in aw.lib.awsrc_last_error_message()


def test_noalloc_decode_f32_and_header_count_pf_stream():
    """F32 weights decoded in place, and a progressive AWSRC-P_F stream decoded
    with K = -1 (the header's record count, read on the device), each against
    the regular dense decoder, twice in a row."""
    import paper_2608_23144_gb300 as aw
    cases = [
        (_case(aw, [(72, 256), (40, 64)], 3, w_dtype="f32", C=64, P=4, b=4, S=128), None),
        (_case(aw, [(90, 128), (33, 192)], 4, rates=(0.25, 1.0), C=64, P=4, b=4, S=96, variant=1), -1),
    ]
    for _ in range(2):
        for (mods, prm, stream, K), k_arg in cases:
            k_call = K if k_arg is None else k_arg
            ref = aw.awsrc_decode_apply(prm, mods, stream, k_call, mode=aw.DECODE_DENSE)
            outs = [m["W0"].clone() for m in mods]
            aw.awsrc_decode_apply_inplace_noalloc(prm, mods, stream, k_call, outs)
            torch.cuda.synchronize()
            for a, b in zip(ref, outs):
                assert a.dtype == b.dtype and torch.equal(a, b)
            assert any(not torch.equal(o, m["W0"]) for o, m in zip(outs, mods))
