"""ctypes marshalling around the plain C oracle (``awsrc_oracle.c``).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``). Every function here
converts numpy arrays and forwards to one C function; the arithmetic lives in
the C file, which follows the paper step by step:

* ``gen_basis``         GenBasis of Eq. 2 (Sec. 3.1)
* ``score_candidate``   Eq. 3 fit, Sec. 3.2 quantisation, Eq. 4 gain (binary32)
* ``encode_tiles``      Sec. 3.2 seed search (binary32)
* ``def_fit/def_gain``  Eq. 3 and Eq. 4 in double (definition mode)
* ``select_records``    Sec. 3.3 allocation and Sec. 3.4 serialisation (Eq. 5)
* ``decode_apply``      Sec. 3.2 decoder
* ``rtn_quantize``      the RTN-INT4 g128 backbone (Eq. 1, Sec. 4) and SDQ (Sec. 3.3)
* ``packed_gemv``       (W0 + r_hat) x in double from the packed backbone and a stream
"""
from __future__ import annotations

import ctypes as ct
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "awsrc_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None

CANDIDATE_DTYPE = np.dtype(
    [("gain", "<f4"), ("seed", "<u2"), ("scale", "<i2"), ("code", "i1", (8,))], align=False
)
assert CANDIDATE_DTYPE.itemsize == 16


class Params(ct.Structure):
    _fields_ = [
        ("C", ct.c_int32), ("P", ct.c_int32), ("b", ct.c_int32), ("S", ct.c_int32),
        ("b_e", ct.c_int32), ("e_bias", ct.c_int32),
        ("scale_mode", ct.c_int32), ("permute", ct.c_int32), ("variant", ct.c_int32),
        ("ridge_rel", ct.c_float), ("gen_seed", ct.c_uint64),
    ]


def _source() -> str:
    """The oracle's C source. AWSRC_ORACLE_SRC names another file only for the
    mutation test of the pins, which builds copies of this source with one
    planted mistake each; unset, it is the oracle itself."""
    return os.environ.get("AWSRC_ORACLE_SRC") or _SRC


def build(force: bool = False, src: str = None) -> str:
    """Compile the oracle with gcc (-ffp-contract=off: no implicit fusion)."""
    src = src or _source()
    if src == _SRC:
        os.makedirs(_BUILD, exist_ok=True)
        path = _LIB_PATH
    else:  # a copy built by the mutation test, next to its source
        path = os.path.splitext(src)[0] + ".so"
    if not force and os.path.exists(path) and os.path.getmtime(path) >= os.path.getmtime(src):
        return path
    tmp = path + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=gnu11", "-ffp-contract=off", "-fno-fast-math", "-fopenmp",
           "-fPIC", "-shared", "-o", tmp, src, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, path)
    return path


def lib():
    global _lib
    with _lock:
        if _lib is None:
            L = ct.CDLL(build())
            P = ct.POINTER
            vp = ct.c_void_p
            L.orc_num_threads.restype = ct.c_int
            L.orc_num_threads.argtypes = []
            L.orc_splitmix64_output.restype = ct.c_uint64
            L.orc_splitmix64_output.argtypes = [ct.c_uint64, ct.c_uint64]
            L.orc_gen_basis.argtypes = [ct.c_uint64, ct.c_uint32, ct.c_int, ct.c_int, ct.c_int, vp, vp, vp, vp]
            L.orc_f32_to_f16.restype = ct.c_uint16
            L.orc_f32_to_f16.argtypes = [ct.c_float]
            L.orc_f16_to_f32.restype = ct.c_float
            L.orc_f16_to_f32.argtypes = [ct.c_uint16]
            L.orc_f32_to_bf16.restype = ct.c_uint16
            L.orc_f32_to_bf16.argtypes = [ct.c_float]
            L.orc_fixed_point.restype = ct.c_int
            L.orc_fixed_point.argtypes = [ct.c_int, vp, vp]
            L.orc_tile_valid.restype = ct.c_int
            L.orc_tile_valid.argtypes = [ct.c_int, vp, vp]
            L.orc_score_candidate.restype = ct.c_int
            L.orc_score_candidate.argtypes = [P(Params), vp, vp, vp, vp, vp, vp, vp]
            L.orc_encode_tiles.argtypes = [P(Params), ct.c_int64, ct.c_int64, vp, vp, vp, vp,
                                           ct.c_float, ct.c_float, vp, ct.c_int64, ct.c_int64, vp]
            L.orc_encode_tile_list.argtypes = [P(Params), ct.c_int64, ct.c_int64, vp, vp, vp, vp,
                                               ct.c_float, ct.c_float, vp, vp, ct.c_int64, vp]
            L.orc_def_fit.restype = ct.c_int
            L.orc_def_fit.argtypes = [ct.c_int, ct.c_int, ct.c_double, vp, vp, vp, vp]
            L.orc_def_gain.restype = ct.c_double
            L.orc_def_gain.argtypes = [ct.c_int, ct.c_int, vp, vp, vp, vp, ct.c_double]
            L.orc_header_bytes.restype = ct.c_int64
            L.orc_header_bytes.argtypes = [ct.c_int32]
            L.orc_record_bytes.restype = ct.c_int64
            L.orc_record_bytes.argtypes = [P(Params), ct.c_int64]
            L.orc_budget_bytes.restype = ct.c_int64
            L.orc_budget_bytes.argtypes = [ct.c_double, ct.c_int64]
            L.orc_pack_record.argtypes = [P(Params), ct.c_int64, ct.c_int64, vp, vp]
            L.orc_unpack_record.argtypes = [P(Params), ct.c_int64, vp, vp, vp]
            L.orc_select_records.restype = ct.c_int
            L.orc_select_records.argtypes = [P(Params), ct.c_int32, vp, vp, vp, vp, ct.c_int32,
                                             vp, ct.c_int64, vp, vp]
            L.orc_decode_apply.restype = ct.c_int
            L.orc_decode_apply.argtypes = [P(Params), ct.c_int32, vp, vp, vp, ct.c_int64, vp, ct.c_int]
            L.orc_rtn_quantize.argtypes = [ct.c_int64, ct.c_int64, ct.c_int, ct.c_int, ct.c_int, vp, vp, vp, vp,
                                           vp, vp, vp]
            L.orc_packed_gemv.restype = ct.c_int
            L.orc_packed_gemv.argtypes = [P(Params), ct.c_int32, vp, vp, ct.c_int32, ct.c_int, vp, vp, vp,
                                          ct.c_int64, ct.c_int, vp, vp, vp]
            _lib = L
    return _lib


def params(C=64, P=4, b=4, S=256, b_e=8, e_bias=0, scale_mode=0, permute=1, variant=0,
           ridge_rel=1e-6, gen_seed=0) -> Params:
    return Params(C, P, b, S, b_e, e_bias, scale_mode, permute, variant,
                  ct.c_float(ridge_rel).value, gen_seed)


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ct.c_void_p)


def num_threads() -> int:
    return int(lib().orc_num_threads())


def splitmix64_output(x: int, n: int) -> int:
    return int(lib().orc_splitmix64_output(x, n))


def gen_basis(gen_seed: int, s: int, C: int, P: int, permute: int = 1):
    """GenBasis (Eq. 2): returns sign[C], perm[C], cols[P], negmask[P, C] (1 = negative)."""
    sign = np.zeros(C, np.uint8)
    perm = np.zeros(C, np.int32)
    cols = np.zeros(P, np.int32)
    neg = np.zeros((P, C), np.uint8)
    lib().orc_gen_basis(gen_seed, s, C, P, permute, _ptr(sign), _ptr(perm), _ptr(cols), _ptr(neg))
    return sign, perm, cols, neg


def basis_masks(prm: Params) -> np.ndarray:
    """negmask for every seed: uint8[S, P, C]."""
    out = np.zeros((prm.S, prm.P, prm.C), np.uint8)
    for s in range(prm.S):
        out[s] = gen_basis(prm.gen_seed, s, prm.C, prm.P, prm.permute)[3]
    return out


def basis_matrix(gen_seed: int, s: int, C: int, P: int, permute: int = 1) -> np.ndarray:
    """B_s as a float64 C x P matrix with entries +-C^-1/2."""
    neg = gen_basis(gen_seed, s, C, P, permute)[3]
    return np.where(neg.T == 1, -1.0, 1.0) / np.sqrt(C)


def f32_to_f16_bits(x: float) -> int:
    return int(lib().orc_f32_to_f16(ct.c_float(x)))


def f16_bits_to_f32(h: int) -> float:
    return float(lib().orc_f16_to_f32(h))


def f32_to_bf16_bits(x: float) -> int:
    return int(lib().orc_f32_to_bf16(ct.c_float(x)))


def score_candidate(prm: Params, r, d, negmask):
    """Spec-mode score of one (tile, seed). Returns dict or None when invalid."""
    r = np.ascontiguousarray(r, np.float32)
    d = np.ascontiguousarray(d, np.float32)
    neg = np.ascontiguousarray(negmask, np.uint8)
    g = np.zeros(1, np.float32)
    sf = np.zeros(1, np.int16)
    codes = np.zeros(8, np.int8)
    alpha = np.zeros(8, np.float32)
    ok = lib().orc_score_candidate(ct.byref(prm), _ptr(r), _ptr(d), _ptr(neg), _ptr(g), _ptr(sf),
                                   _ptr(codes), _ptr(alpha))
    if not ok:
        return None
    return {"gain": float(g[0]), "scale": int(sf[0]), "codes": codes[: prm.P].astype(np.int64),
            "alpha": alpha[: prm.P].copy()}


def fixed_point(x):
    """Per-tile fixed point of the correlations: returns (q, X) with X = rint(x 2^-q)."""
    x = np.ascontiguousarray(x, np.float32)
    X = np.zeros(len(x), np.int32)
    q = lib().orc_fixed_point(len(x), _ptr(x), _ptr(X))
    return int(q), X


def tile_valid(r, d) -> bool:
    r = np.ascontiguousarray(r, np.float32)
    d = np.ascontiguousarray(d, np.float32)
    return bool(lib().orc_tile_valid(len(r), _ptr(r), _ptr(d)))


def _as_f32(a):
    return None if a is None else np.ascontiguousarray(a, np.float32)


def encode_tiles(prm: Params, W, W0, act, fisher=None, w_act=1.0, w_fisher=0.0, tiles=None,
                 masks=None) -> np.ndarray:
    """Spec-mode seed search (Sec. 3.2) for one module; W/W0 are float arrays
    (bfloat16 inputs widened exactly). tiles: None = all, else an index array."""
    W = _as_f32(W)
    W0 = _as_f32(W0)
    act = _as_f32(act)
    fisher = _as_f32(fisher)
    rows, cols = W.shape
    if masks is None:
        masks = basis_masks(prm)
    masks = np.ascontiguousarray(masks, np.uint8)
    if prm.variant == 1 and (fisher is None or fisher.shape != W.shape):
        raise ValueError("the PF variant needs a Fisher diagonal of the module's shape")
    fptr = _ptr(fisher) if fisher is not None else None
    if tiles is None:
        T = rows * cols // prm.C
        out = np.zeros(T, CANDIDATE_DTYPE)
        lib().orc_encode_tiles(ct.byref(prm), rows, cols, _ptr(W), _ptr(W0), _ptr(act), fptr,
                               ct.c_float(w_act), ct.c_float(w_fisher), _ptr(masks), 0, T, _ptr(out))
    else:
        tiles = np.ascontiguousarray(tiles, np.int64)
        out = np.zeros(len(tiles), CANDIDATE_DTYPE)
        lib().orc_encode_tile_list(ct.byref(prm), rows, cols, _ptr(W), _ptr(W0), _ptr(act), fptr,
                                   ct.c_float(w_act), ct.c_float(w_fisher), _ptr(masks),
                                   _ptr(tiles), len(tiles), _ptr(out))
    return out


def def_fit(C, P, ridge_rel, r, d, negmask):
    """Definition mode Eq. 3 (double, Gaussian elimination)."""
    r = np.ascontiguousarray(r, np.float64)
    d = np.ascontiguousarray(d, np.float64)
    neg = np.ascontiguousarray(negmask, np.uint8)
    alpha = np.zeros(P, np.float64)
    ok = lib().orc_def_fit(C, P, float(ridge_rel), _ptr(r), _ptr(d), _ptr(neg), _ptr(alpha))
    return alpha if ok else None


def def_gain(C, P, r, d, negmask, codes, scale) -> float:
    """Definition mode Eq. 4 numerator (double, direct from the reconstruction)."""
    r = np.ascontiguousarray(r, np.float64)
    d = np.ascontiguousarray(d, np.float64)
    neg = np.ascontiguousarray(negmask, np.uint8)
    codes = np.ascontiguousarray(codes, np.int32)
    return float(lib().orc_def_gain(C, P, _ptr(r), _ptr(d), _ptr(neg), _ptr(codes), float(scale)))


def scale_value(prm: Params, scale_field: int) -> float:
    """The float scale a candidate's scale field stands for."""
    if prm.scale_mode == 0:
        return float(np.ldexp(np.float32(1.0), int(scale_field)))
    return f16_bits_to_f32(int(scale_field) & 0xFFFF)


def header_bytes(n_mod: int) -> int:
    return int(lib().orc_header_bytes(n_mod))


def record_bytes(prm: Params, T: int) -> int:
    return int(lib().orc_record_bytes(ct.byref(prm), T))


def budget_bytes(rate: float, n_scope: int) -> int:
    return int(lib().orc_budget_bytes(rate, n_scope))


def pack_record(prm: Params, T: int, tile: int, cand) -> bytes:
    L = record_bytes(prm, T)
    rec = np.zeros(L, np.uint8)
    c = np.zeros(1, CANDIDATE_DTYPE)
    c[0] = cand
    lib().orc_pack_record(ct.byref(prm), T, tile, _ptr(c), _ptr(rec))
    return rec.tobytes()


def unpack_record(prm: Params, T: int, rec: bytes):
    buf = np.frombuffer(rec, np.uint8).copy()
    tile = np.zeros(1, np.int64)
    c = np.zeros(1, CANDIDATE_DTYPE)
    lib().orc_unpack_record(ct.byref(prm), T, _ptr(buf), _ptr(tile), _ptr(c))
    return int(tile[0]), c[0]


def select_records(prm: Params, shapes, cands: np.ndarray, rates):
    """Sec. 3.3 allocation + Sec. 3.4 serialisation. shapes: [(rows, cols)] per module,
    cands: CANDIDATE_DTYPE over all modules' tiles (global order).
    Returns (stream bytes, counts, bytes_per_rate)."""
    n_mod = len(shapes)
    mod_tiles = np.array([r * c // prm.C for r, c in shapes], np.int64)
    mod_w = np.array([r * c for r, c in shapes], np.int64)
    rates = np.ascontiguousarray(rates, np.float64)
    T = int(mod_tiles.sum())
    cands = np.ascontiguousarray(cands, CANDIDATE_DTYPE)
    assert len(cands) == T
    cap = header_bytes(n_mod) + T * record_bytes(prm, T)
    stream = np.zeros(cap, np.uint8)
    counts = np.zeros(max(n_mod, len(rates)), np.int64)
    nbytes = np.zeros(len(rates), np.int64)
    rc = lib().orc_select_records(ct.byref(prm), n_mod, _ptr(mod_tiles), _ptr(mod_w), _ptr(cands),
                                  _ptr(rates), len(rates), _ptr(stream), cap, _ptr(counts), _ptr(nbytes))
    if rc != 0:
        raise ValueError(f"oracle select_records failed with status {rc}")
    total = int(nbytes.max())
    ncount = n_mod if prm.variant == 0 else len(rates)
    return stream[:total].tobytes(), counts[:ncount].copy(), nbytes.copy()


def decode_apply(prm: Params, W0_list, stream: bytes, K: int, out_bf16: bool = False):
    """Sec. 3.2 decoder on float copies of W0. Returns (list of arrays, bad_flag)."""
    outs = [np.array(w, np.float32, copy=True, order="C") for w in W0_list]
    rows = np.array([o.shape[0] for o in outs], np.int64)
    cols = np.array([o.shape[1] for o in outs], np.int64)
    ptrs = (ct.c_void_p * len(outs))(*[o.ctypes.data for o in outs])
    buf = np.frombuffer(stream, np.uint8).copy()
    bad = lib().orc_decode_apply(ct.byref(prm), len(outs), _ptr(rows), _ptr(cols), _ptr(buf), K,
                                 ptrs, int(out_bf16))
    return outs, int(bad)


def rtn_quantize(W, group: int = 128, sdq: bool = False, block: int = 256):
    """RTN-INT4 backbone and optional scale double quantisation of one module.
    Returns dict(q, s16, c8, consts, s_eff, W0) (W0 in float32)."""
    W = np.ascontiguousarray(W, np.float32)
    rows, cols = W.shape
    assert cols % group == 0
    G = rows * cols // group
    nb = (G + block - 1) // block
    q = np.zeros((rows, cols), np.int8)
    s16 = np.zeros(G, np.uint16)
    c8 = np.zeros(G, np.int8)
    consts = np.zeros(2 * nb, np.float32)
    s_eff = np.zeros(G, np.float32)
    W0 = np.zeros((rows, cols), np.float32)
    lib().orc_rtn_quantize(ct.c_int64(rows), ct.c_int64(cols), group, int(sdq), block, _ptr(W), _ptr(q),
                           _ptr(s16), _ptr(c8), _ptr(consts), _ptr(s_eff), _ptr(W0))
    return {"q": q, "s16": s16, "c8": c8, "consts": consts, "s_eff": s_eff, "W0": W0}


def packed_gemv(prm: Params, q, s_eff, group: int, stream: bytes, K: int, x, shapes=None, m: int = 0):
    """y = (W0 + r_hat) x in double for module m of a stream over `shapes`
    (default: the one module of q). Returns (y, yabs, bad): y and yabs of
    shape (M, rows), yabs = sum_j |(W0 + r_hat)_ij x_j|."""
    q = np.ascontiguousarray(q, np.int8)
    rows, cols = q.shape
    if shapes is None:
        shapes = [(rows, cols)]
    assert tuple(shapes[m]) == (rows, cols)
    mr = np.array([r for r, _ in shapes], np.int64)
    mc = np.array([c for _, c in shapes], np.int64)
    x = np.ascontiguousarray(np.atleast_2d(x), np.float32)
    M = x.shape[0]
    y = np.zeros((M, rows), np.float64)
    yabs = np.zeros((M, rows), np.float64)
    buf = np.frombuffer(stream, np.uint8).copy()
    bad = lib().orc_packed_gemv(ct.byref(prm), len(shapes), _ptr(mr), _ptr(mc), m, group, _ptr(q),
                                _ptr(np.ascontiguousarray(s_eff, np.float32)), _ptr(buf), ct.c_int64(K), M,
                                _ptr(x), _ptr(y), _ptr(yabs))
    return y, yabs, int(bad)
