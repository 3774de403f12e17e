"""ctypes binding of libawsrc.so (include/awsrc.h): argument marshalling only.

Every entry point takes torch tensors that already live on the current CUDA
device, passes their data pointers and the current stream to the C ABI and
returns the output tensors. Workspaces are allocated here, on the caller's
side of the ABI, with torch's allocator; the library itself allocates nothing.
If the shared library is missing the import of this module fails loudly: there
is no CPU fallback.
"""
from __future__ import annotations

import ctypes as ct
import os
from typing import Dict, List, Optional, Sequence

import numpy as np
import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libawsrc.so")

VARIANT_U, VARIANT_PF = 0, 1
SCALE_POW2, SCALE_FP16 = 0, 1
DTYPE_F32, DTYPE_BF16 = 0, 1
DECODE_DENSE, DECODE_INPLACE = 0, 1

STATUS = {0: "ok", 1: "invalid argument", 2: "shape", 3: "unsupported", 4: "budget",
          5: "cuda", 6: "workspace", 7: "capacity", 8: "device fault"}

CANDIDATE_DTYPE = np.dtype([("gain", "<f4"), ("seed", "<u2"), ("scale", "<i2"), ("code", "i1", (8,))])


class AwsrcError(RuntimeError):
    def __init__(self, status: int, where: str, msg: str = ""):
        super().__init__(f"{where}: awsrc status {status} ({STATUS.get(status, '?')}) {msg}".strip())
        self.status = status


class Params(ct.Structure):
    _fields_ = [
        ("C", ct.c_int32), ("P", ct.c_int32), ("b", ct.c_int32), ("S", ct.c_int32),
        ("b_e", ct.c_int32), ("e_bias", ct.c_int32),
        ("scale_mode", ct.c_int32), ("permute", ct.c_int32), ("variant", ct.c_int32),
        ("ridge_rel", ct.c_float), ("gen_seed", ct.c_uint64),
    ]


class Module(ct.Structure):
    _fields_ = [
        ("rows", ct.c_int64), ("cols", ct.c_int64),
        ("w_dtype", ct.c_int32), ("w0_dtype", ct.c_int32),
        ("W", ct.c_void_p), ("W0", ct.c_void_p),
        ("act", ct.c_void_p), ("fisher", ct.c_void_p),
        ("w_act", ct.c_float), ("w_fisher", ct.c_float),
    ]


class PackedWeights(ct.Structure):
    _fields_ = [("codes", ct.c_void_p), ("scales", ct.c_void_p), ("sdq_codes", ct.c_void_p),
                ("sdq_consts", ct.c_void_p), ("sdq", ct.c_int32), ("pad_", ct.c_int32)]


class RtnTask(ct.Structure):
    _fields_ = [("rows", ct.c_int64), ("cols", ct.c_int64), ("W", ct.c_void_p), ("w_dtype", ct.c_int32),
                ("sdq", ct.c_int32), ("codes", ct.c_void_p), ("scales", ct.c_void_p), ("sdq_codes", ct.c_void_p),
                ("sdq_consts", ct.c_void_p), ("W0", ct.c_void_p), ("w0_dtype", ct.c_int32), ("pad_", ct.c_int32)]


class GemvTask(ct.Structure):
    _fields_ = [("m", ct.c_int32), ("pad_", ct.c_int32), ("pw", PackedWeights), ("x", ct.c_void_p),
                ("y", ct.c_void_p)]


def params(C=64, P=4, b=4, S=4096, b_e=8, e_bias=0, scale_mode=SCALE_POW2, permute=1,
           variant=VARIANT_U, ridge_rel=1e-6, gen_seed=0) -> Params:
    return Params(C, P, b, S, b_e, e_bias, scale_mode, permute, variant,
                  ct.c_float(ridge_rel).value, gen_seed)


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(
            f"AWSRC CUDA library not built ({LIB_PATH} missing): run "
            "`python -c 'import __graft_entry__ as g; g.build()'` first")
    L = ct.CDLL(LIB_PATH)
    P = ct.POINTER
    vp, sz = ct.c_void_p, ct.c_size_t
    st = ct.c_int
    L.awsrc_status_string.restype = ct.c_char_p
    L.awsrc_status_string.argtypes = [st]
    L.awsrc_last_error_message.restype = ct.c_char_p
    L.awsrc_last_error_message.argtypes = []
    L.awsrc_record_bytes.restype = ct.c_int64
    L.awsrc_record_bytes.argtypes = [P(Params), ct.c_int64]
    L.awsrc_header_bytes.restype = ct.c_int64
    L.awsrc_header_bytes.argtypes = [ct.c_int32]
    L.awsrc_encode_workspace_bytes.restype = st
    L.awsrc_encode_workspace_bytes.argtypes = [P(Params), ct.c_int32, P(Module), P(sz)]
    L.awsrc_encode_tiles.restype = st
    L.awsrc_encode_tiles.argtypes = [P(Params), ct.c_int32, P(Module), vp, vp, sz, vp]
    L.awsrc_gen_basis.restype = st
    L.awsrc_gen_basis.argtypes = [P(Params), vp, vp]
    L.awsrc_stream_capacity.restype = st
    L.awsrc_stream_capacity.argtypes = [P(Params), ct.c_int32, P(Module), P(ct.c_double), ct.c_int32, P(sz)]
    L.awsrc_select_workspace_bytes.restype = st
    L.awsrc_select_workspace_bytes.argtypes = [P(Params), ct.c_int32, P(Module), P(sz)]
    L.awsrc_select_records.restype = st
    L.awsrc_select_records.argtypes = [P(Params), ct.c_int32, P(Module), vp, P(ct.c_double), ct.c_int32,
                                       vp, sz, vp, vp, vp, sz, vp]
    L.awsrc_decode_workspace_bytes.restype = st
    L.awsrc_decode_workspace_bytes.argtypes = [P(Params), ct.c_int32, P(Module), ct.c_int32, P(sz)]
    L.awsrc_decode_apply.restype = st
    L.awsrc_decode_apply.argtypes = [P(Params), ct.c_int32, P(Module), vp, sz, ct.c_int64, P(vp), ct.c_int32,
                                     ct.c_int32, vp, sz, vp]
    L.awsrc_decode_apply_inplace_noalloc.restype = st
    L.awsrc_decode_apply_inplace_noalloc.argtypes = [P(Params), ct.c_int32, P(Module), vp, sz, ct.c_int64,
                                                     P(vp), vp]
    L.awsrc_set_timing_events.restype = None
    L.awsrc_set_timing_events.argtypes = [vp, vp]
    L.awsrc_kernel_launches.restype = ct.c_uint64
    L.awsrc_kernel_launches.argtypes = []
    L.awsrc_set_search_pruning.restype = None
    L.awsrc_set_search_pruning.argtypes = [ct.c_int32]
    L.awsrc_set_wait_test.restype = None
    L.awsrc_set_wait_test.argtypes = [ct.c_uint64, ct.c_int32]
    L.awsrc_verify_reciprocal.restype = st
    L.awsrc_verify_reciprocal.argtypes = [ct.c_uint32, ct.c_uint32, vp, vp]
    L.awsrc_workspace_status.restype = st
    L.awsrc_workspace_status.argtypes = [vp, vp, P(ct.c_uint32)]
    L.awsrc_rtn_quantize.restype = st
    L.awsrc_rtn_quantize.argtypes = [ct.c_int64, ct.c_int64, vp, ct.c_int32, ct.c_int32, vp, vp, vp, vp, vp,
                                     ct.c_int32, vp]
    L.awsrc_rtn_quantize_batch.restype = st
    L.awsrc_rtn_quantize_batch.argtypes = [ct.c_int32, P(RtnTask), vp]
    L.awsrc_backbone_metadata_bytes.restype = ct.c_int64
    L.awsrc_backbone_metadata_bytes.argtypes = [ct.c_int64, ct.c_int64, ct.c_int32]
    L.awsrc_rate_with_sdq_savings.restype = st
    L.awsrc_rate_with_sdq_savings.argtypes = [ct.c_int32, P(Module), ct.c_double, P(ct.c_double),
                                              P(ct.c_int64)]
    L.awsrc_sidecar_workspace_bytes.restype = st
    L.awsrc_sidecar_workspace_bytes.argtypes = [P(Params), ct.c_int32, P(Module), P(sz)]
    L.awsrc_sidecar_prepare.restype = st
    L.awsrc_sidecar_prepare.argtypes = [P(Params), ct.c_int32, P(Module), vp, sz, ct.c_int64, vp, sz, vp]
    L.awsrc_packed_gemv.restype = st
    L.awsrc_packed_gemv.argtypes = [P(Params), ct.c_int32, P(Module), ct.c_int32, P(PackedWeights), vp, sz,
                                    ct.c_int32, vp, vp, vp]
    L.awsrc_packed_gemv_batch.restype = st
    L.awsrc_packed_gemv_batch.argtypes = [P(Params), ct.c_int32, P(Module), ct.c_int32, P(GemvTask), vp, sz,
                                          ct.c_int32, vp]
    return L


lib = _load()


def _check(status: int, where: str):
    if status != 0:
        msg = lib.awsrc_last_error_message().decode() if status == 5 else ""
        raise AwsrcError(status, where, msg)


def _stream(stream=None) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return DTYPE_F32
    if t.dtype == torch.bfloat16:
        return DTYPE_BF16
    raise TypeError(f"unsupported weight dtype {t.dtype} (float32 or bfloat16)")


def _dev_ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    if t is None:
        return None
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError("tensors passed to the AWSRC library must be contiguous CUDA tensors")
    return t.data_ptr()


def _require(t, name: str, dtype=None, shape=None, numel: Optional[int] = None, device=None):
    """Check a tensor argument on the host before its pointer crosses the ABI.
    The kernels index every array by the module shapes they are given, so a
    tensor that is smaller, of another element type or on another device than
    those shapes imply would be read or written out of bounds on the device."""
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor, not {type(t).__name__}")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, not {t.dtype}")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")
    if numel is not None and t.numel() < numel:
        raise ValueError(f"{name} holds {t.numel()} elements, at least {numel} are needed")
    if device is not None and t.device != device:
        raise ValueError(f"{name} is on {t.device}, expected {device}")


def _shape(m: Dict[str, object], i: int):
    """(rows, cols) of module i, from its W0."""
    W0 = m["W0"]
    _require(W0, f"modules[{i}]['W0']")
    if W0.dim() != 2:
        raise ValueError(f"modules[{i}]['W0'] must be 2-D (rows x cols), not {W0.dim()}-D")
    return int(W0.shape[0]), int(W0.shape[1])


def module_array(modules: Sequence[Dict[str, object]], decoder: bool = False):
    """awsrc_module[] from dicts with W, W0, act (and fisher, w_act, w_fisher).
    W must have W0's shape, act is float32 with cols entries and fisher float32
    rows x cols, all on W0's device."""
    arr = (Module * len(modules))()
    for i, m in enumerate(modules):
        W0 = m["W0"]
        W = m.get("W")
        rows, cols = _shape(m, i)
        dev = W0.device
        if not decoder:
            if W is not None:
                _require(W, f"modules[{i}]['W']", shape=(rows, cols), device=dev)
            if m.get("act") is not None:
                _require(m["act"], f"modules[{i}]['act']", dtype=torch.float32, numel=cols, device=dev)
            if m.get("fisher") is not None:
                _require(m["fisher"], f"modules[{i}]['fisher']", dtype=torch.float32, shape=(rows, cols),
                         device=dev)
        arr[i].rows, arr[i].cols = rows, cols
        arr[i].w0_dtype = _dtype_code(W0)
        arr[i].W0 = _dev_ptr(W0)
        if W is not None and not decoder:
            arr[i].w_dtype = _dtype_code(W)
            arr[i].W = _dev_ptr(W)
        if m.get("act") is not None and not decoder:
            arr[i].act = _dev_ptr(m["act"])
        if m.get("fisher") is not None and not decoder:
            arr[i].fisher = _dev_ptr(m["fisher"])
        arr[i].w_act = float(m.get("w_act", 1.0))
        arr[i].w_fisher = float(m.get("w_fisher", 0.0))
    return arr


def _tiles(prm: Params, modules) -> int:
    return sum(r * c // prm.C for r, c in (_shape(m, i) for i, m in enumerate(modules)))


def awsrc_record_bytes(prm: Params, T: int) -> int:
    return int(lib.awsrc_record_bytes(ct.byref(prm), T))


def awsrc_header_bytes(n_mod: int) -> int:
    return int(lib.awsrc_header_bytes(n_mod))


def awsrc_encode_workspace_bytes(prm: Params, modules) -> int:
    mods = module_array(modules)
    n = ct.c_size_t()
    _check(lib.awsrc_encode_workspace_bytes(ct.byref(prm), len(modules), mods, ct.byref(n)), "encode_workspace_bytes")
    return n.value


def awsrc_encode_tiles(prm: Params, modules, out: Optional[torch.Tensor] = None,
                       workspace: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """Seed search (Sec. 3.2): one best candidate per tile, uint8 [T, 16] on the device."""
    T = _tiles(prm, modules)
    dev = modules[0]["W0"].device
    if out is None:
        out = torch.empty((T, 16), dtype=torch.uint8, device=dev)
    _require(out, "out", dtype=torch.uint8, numel=16 * T, device=dev)
    mods = module_array(modules)
    need = awsrc_encode_workspace_bytes(prm, modules)
    if workspace is None or workspace.numel() < need:
        workspace = torch.empty(need, dtype=torch.uint8, device=dev)
    _check(lib.awsrc_encode_tiles(ct.byref(prm), len(modules), mods, _dev_ptr(out), _dev_ptr(workspace),
                                  workspace.numel(), _stream(stream)), "encode_tiles")
    out._awsrc_workspace = workspace  # keep alive for awsrc_workspace_status
    return out


def _rtn_buffers(W: torch.Tensor, sdq: bool, w0_dtype, out: Optional[Dict[str, torch.Tensor]]):
    """Checks W (and `out`, when given) or allocates the outputs of one module."""
    _require(W, "W")
    if W.dim() != 2:
        raise ValueError(f"W must be 2-D (rows x cols), not {W.dim()}-D")
    rows, cols = W.shape
    dev = W.device
    G = rows * cols // 128
    if out is not None:  # buffers of an earlier call: the same shape and SDQ setting
        _require(out["codes"], "out['codes']", dtype=torch.uint8, numel=rows * cols // 2, device=dev)
        _require(out["scales"], "out['scales']", dtype=torch.int16, numel=G, device=dev)
        _require(out["W0"], "out['W0']", shape=(rows, cols), device=dev)
        if sdq:
            _require(out["sdq_codes"], "out['sdq_codes']", dtype=torch.int8, numel=G, device=dev)
            _require(out["sdq_consts"], "out['sdq_consts']", dtype=torch.float32, numel=2 * ((G + 255) // 256),
                     device=dev)
        return out
    out = {"codes": torch.empty(rows * cols // 2, dtype=torch.uint8, device=dev),
           "scales": torch.empty(G, dtype=torch.int16, device=dev)}
    if sdq:
        out["sdq_codes"] = torch.empty(G, dtype=torch.int8, device=dev)
        out["sdq_consts"] = torch.empty(2 * ((G + 255) // 256), dtype=torch.float32, device=dev)
    w0t = W.dtype if w0_dtype is None else w0_dtype
    out["W0"] = torch.empty(rows, cols, dtype=w0t, device=dev)
    return out


def awsrc_rtn_quantize(W: torch.Tensor, sdq: bool = False, w0_dtype=None, stream=None,
                       out: Optional[Dict[str, torch.Tensor]] = None) -> Dict[str, torch.Tensor]:
    """RTN-INT4 backbone of one module (groups of 128 inputs), optional SDQ.
    Returns codes (uint8, two per byte), scales (binary16 bits as int16),
    sdq_codes (int8) and sdq_consts (float32 mean, step per 256 groups) when
    sdq, and W0 (in w0_dtype, default W's dtype). `out` reuses the buffers of
    an earlier call on the same shape."""
    out = _rtn_buffers(W, sdq, w0_dtype, out)
    rows, cols = W.shape
    _check(lib.awsrc_rtn_quantize(rows, cols, _dev_ptr(W), _dtype_code(W), int(sdq), _dev_ptr(out["codes"]),
                                  _dev_ptr(out["scales"]), _dev_ptr(out.get("sdq_codes")),
                                  _dev_ptr(out.get("sdq_consts")), _dev_ptr(out["W0"]), _dtype_code(out["W0"]),
                                  _stream(stream)), "rtn_quantize")
    return out


def awsrc_rtn_quantize_batch(Ws: Sequence[torch.Tensor], sdq: bool = False, w0_dtype=None, stream=None,
                             outs: Optional[List[Dict[str, torch.Tensor]]] = None) -> List[Dict[str, torch.Tensor]]:
    """awsrc_rtn_quantize of several modules in one launch (per run of equal
    dtypes); returns one output dict per module, as the single call does."""
    if outs is not None and len(outs) != len(Ws):
        raise ValueError(f"{len(outs)} output sets for {len(Ws)} modules")
    res = [_rtn_buffers(W, sdq, w0_dtype, None if outs is None else outs[i]) for i, W in enumerate(Ws)]
    arr = (RtnTask * len(Ws))()
    for i, (W, o) in enumerate(zip(Ws, res)):
        arr[i] = RtnTask(W.shape[0], W.shape[1], _dev_ptr(W), _dtype_code(W), int(sdq), _dev_ptr(o["codes"]),
                         _dev_ptr(o["scales"]), _dev_ptr(o.get("sdq_codes")), _dev_ptr(o.get("sdq_consts")),
                         _dev_ptr(o["W0"]), _dtype_code(o["W0"]), 0)
    _check(lib.awsrc_rtn_quantize_batch(len(Ws), arr, _stream(stream)), "rtn_quantize_batch")
    return res


def awsrc_backbone_metadata_bytes(rows: int, cols: int, sdq: bool) -> int:
    return int(lib.awsrc_backbone_metadata_bytes(rows, cols, int(sdq)))


def awsrc_rate_with_sdq_savings(shapes, rate: float):
    """(rate for awsrc_select_records, saved bytes): the sidecar budget grows by
    the metadata bytes SDQ saves on these (rows, cols) modules (Sec. 3.3)."""
    mods = shape_modules(shapes)
    out = ct.c_double()
    saved = ct.c_int64()
    _check(lib.awsrc_rate_with_sdq_savings(len(shapes), mods, float(rate), ct.byref(out), ct.byref(saved)),
           "rate_with_sdq_savings")
    return out.value, saved.value


def shape_modules(shapes):
    """awsrc_module[] carrying only shapes (serving calls read no weights)."""
    arr = (Module * len(shapes))()
    for i, (r, c) in enumerate(shapes):
        arr[i].rows, arr[i].cols = r, c
        arr[i].w0_dtype = DTYPE_BF16
    return arr


def awsrc_sidecar_prepare(prm: Params, shapes, stream_bytes: torch.Tensor, K: int = -1,
                          workspace: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """Unpack a stream once for serving; returns the prepared sidecar workspace."""
    mods = shape_modules(shapes)
    n = ct.c_size_t()
    _check(lib.awsrc_sidecar_workspace_bytes(ct.byref(prm), len(shapes), mods, ct.byref(n)), "sidecar_workspace_bytes")
    if workspace is None or workspace.numel() < n.value:
        workspace = torch.empty(n.value, dtype=torch.uint8, device=stream_bytes.device)
    _check(lib.awsrc_sidecar_prepare(ct.byref(prm), len(shapes), mods, _dev_ptr(stream_bytes), stream_bytes.numel(),
                                     K, _dev_ptr(workspace), workspace.numel(), _stream(stream)), "sidecar_prepare")
    return workspace


def _gemv_operands(shapes, m: int, backbone: Dict[str, torch.Tensor], x: torch.Tensor,
                   y: Optional[torch.Tensor]):
    """Checks one product's operands; returns (x as M x cols, y, PackedWeights)."""
    rows, cols = shapes[m]
    _require(x, "x", dtype=torch.float32)
    if x.numel() % cols != 0:
        raise ValueError(f"x holds {x.numel()} elements, not a whole number of rows of {cols}")
    x = x.reshape(-1, cols)
    dev = x.device
    if y is None:
        y = torch.empty(x.shape[0], rows, dtype=torch.float32, device=dev)
    _require(y, "y", dtype=torch.float32, shape=(x.shape[0], rows), device=dev)
    sdq = "sdq_codes" in backbone
    G = rows * cols // 128
    _require(backbone["codes"], "backbone['codes']", dtype=torch.uint8, numel=rows * cols // 2, device=dev)
    if sdq:
        _require(backbone["sdq_codes"], "backbone['sdq_codes']", dtype=torch.int8, numel=G, device=dev)
        _require(backbone["sdq_consts"], "backbone['sdq_consts']", dtype=torch.float32,
                 numel=2 * ((G + 255) // 256), device=dev)
    else:
        _require(backbone["scales"], "backbone['scales']", dtype=torch.int16, numel=G, device=dev)
    pw = PackedWeights(_dev_ptr(backbone["codes"]), None if sdq else _dev_ptr(backbone["scales"]),
                       _dev_ptr(backbone.get("sdq_codes")), _dev_ptr(backbone.get("sdq_consts")), int(sdq), 0)
    return x, y, pw


def awsrc_packed_gemv(prm: Params, shapes, m: int, backbone: Dict[str, torch.Tensor], x: torch.Tensor,
                      sidecar: Optional[torch.Tensor] = None, y: Optional[torch.Tensor] = None,
                      stream=None) -> torch.Tensor:
    """y = (W0 + r_hat) x for module m (x: M x cols float32); backbone holds
    awsrc_rtn_quantize's codes and scales (or SDQ codes and constants)."""
    mods = shape_modules(shapes)
    _require(x, "x", dtype=torch.float32)
    if sidecar is not None:
        _require(sidecar, "sidecar", dtype=torch.uint8, device=x.device)
    x, y, pw = _gemv_operands(shapes, m, backbone, x, y)
    _check(lib.awsrc_packed_gemv(ct.byref(prm), len(shapes), mods, m, ct.byref(pw), _dev_ptr(sidecar),
                                 0 if sidecar is None else sidecar.numel(), x.shape[0], _dev_ptr(x), _dev_ptr(y),
                                 _stream(stream)), "packed_gemv")
    return y


def awsrc_packed_gemv_batch(prm: Params, shapes, tasks, sidecar: Optional[torch.Tensor] = None,
                            stream=None) -> List[torch.Tensor]:
    """Several products in one launch: tasks is a list of (m, backbone, x) or
    (m, backbone, x, y) with the same number M of vectors; returns the y's."""
    mods = shape_modules(shapes)
    if sidecar is not None and tasks:
        _require(tasks[0][2], "x", dtype=torch.float32)
        _require(sidecar, "sidecar", dtype=torch.uint8, device=tasks[0][2].device)
    arr = (GemvTask * len(tasks))()
    ys, Ms, dev = [], set(), None
    for i, t in enumerate(tasks):
        m, backbone, x = t[0], t[1], t[2]
        x, y, pw = _gemv_operands(shapes, m, backbone, x, t[3] if len(t) > 3 else None)
        if dev is not None and x.device != dev:
            raise ValueError("every task's tensors must be on one device")
        dev = x.device
        Ms.add(x.shape[0])
        arr[i] = GemvTask(m, 0, pw, _dev_ptr(x), _dev_ptr(y))
        ys.append((x, y))  # x kept alive with y until the call returns
    if len(Ms) != 1:
        raise ValueError(f"tasks must share M, got {sorted(Ms)}")
    _check(lib.awsrc_packed_gemv_batch(ct.byref(prm), len(shapes), mods, len(tasks), arr, _dev_ptr(sidecar),
                                       0 if sidecar is None else sidecar.numel(), Ms.pop(), _stream(stream)),
           "packed_gemv_batch")
    return [y for _, y in ys]


def awsrc_gen_basis(prm: Params, stream=None, device="cuda") -> torch.Tensor:
    W = (prm.C + 63) // 64
    masks = torch.empty(prm.S * prm.P * W, dtype=torch.int64, device=device)
    _check(lib.awsrc_gen_basis(ct.byref(prm), _dev_ptr(masks), _stream(stream)), "gen_basis")
    return masks


def awsrc_stream_capacity(prm: Params, modules, rates: Sequence[float]) -> int:
    mods = module_array(modules, decoder=True)
    r = (ct.c_double * len(rates))(*rates)
    n = ct.c_size_t()
    _check(lib.awsrc_stream_capacity(ct.byref(prm), len(modules), mods, r, len(rates), ct.byref(n)), "stream_capacity")
    return n.value


def awsrc_select_records(prm: Params, modules, cands: torch.Tensor, rates: Sequence[float],
                         workspace: Optional[torch.Tensor] = None, stream=None,
                         out: Optional[torch.Tensor] = None, counts: Optional[torch.Tensor] = None,
                         nbytes: Optional[torch.Tensor] = None):
    """Sec. 3.3 allocation + Eq. 5 serialisation. Returns (stream bytes [capacity] uint8,
    counts int64 (U: per module, PF: per rate), bytes int64 (per rate)), all on the device.
    Only the first bytes[r] bytes of the stream are written."""
    _require(cands, "cands", dtype=torch.uint8, numel=16 * _tiles(prm, modules))
    dev = cands.device
    # caller buffers: the stream is bytes, counts and bytes are written as int64
    for name, t, dt in (("out", out, torch.uint8), ("counts", counts, torch.int64), ("nbytes", nbytes, torch.int64)):
        if t is not None:
            _require(t, name, dtype=dt, device=dev)
    mods = module_array(modules, decoder=True)
    r = (ct.c_double * len(rates))(*rates)
    cap = awsrc_stream_capacity(prm, modules, rates)
    n = ct.c_size_t()
    _check(lib.awsrc_select_workspace_bytes(ct.byref(prm), len(modules), mods, ct.byref(n)), "select_workspace_bytes")
    if workspace is None or workspace.numel() < n.value:
        workspace = torch.empty(n.value, dtype=torch.uint8, device=dev)
    if out is None or out.numel() < cap:
        out = torch.zeros(cap, dtype=torch.uint8, device=dev)
    ncount = len(modules) if prm.variant == VARIANT_U else len(rates)
    if counts is None or counts.numel() < ncount:
        counts = torch.empty(ncount, dtype=torch.int64, device=dev)
    if nbytes is None or nbytes.numel() < len(rates):
        nbytes = torch.empty(len(rates), dtype=torch.int64, device=dev)
    _check(lib.awsrc_select_records(ct.byref(prm), len(modules), mods, _dev_ptr(cands), r, len(rates),
                                    _dev_ptr(out), out.numel(), _dev_ptr(counts), _dev_ptr(nbytes),
                                    _dev_ptr(workspace), workspace.numel(), _stream(stream)), "select_records")
    out._awsrc_workspace = workspace
    return out, counts, nbytes


def _check_outs(modules, outs, dtype):
    """One output per module, of the module's shape, in `dtype`, on its device:
    the decoder writes rows*cols elements through each pointer."""
    if len(outs) != len(modules):
        raise ValueError(f"{len(outs)} outputs for {len(modules)} modules")
    for i, (m, o) in enumerate(zip(modules, outs)):
        _require(o, f"outs[{i}]", dtype=dtype, shape=tuple(m["W0"].shape), device=m["W0"].device)


def awsrc_decode_apply(prm: Params, modules, stream_bytes: torch.Tensor, K: int,
                       outs: Optional[List[torch.Tensor]] = None, out_dtype=None,
                       mode: int = DECODE_DENSE, workspace: Optional[torch.Tensor] = None,
                       stream=None) -> List[torch.Tensor]:
    """Decoder (Sec. 3.2): W_hat = W0 + B_s alpha_hat for the first K records (K < 0: all)."""
    dev = stream_bytes.device
    if out_dtype is None:
        out_dtype = outs[0].dtype if outs else modules[0]["W0"].dtype
    if out_dtype not in (torch.float32, torch.bfloat16):
        raise TypeError(f"out_dtype must be torch.float32 or torch.bfloat16, not {out_dtype}")
    code = DTYPE_F32 if out_dtype == torch.float32 else DTYPE_BF16
    if outs is None:
        outs = [torch.empty_like(m["W0"], dtype=out_dtype) for m in modules]
    _check_outs(modules, outs, out_dtype)
    mods = module_array(modules, decoder=True)
    ptrs = (ct.c_void_p * len(outs))(*[_dev_ptr(o) for o in outs])
    n = ct.c_size_t()
    _check(lib.awsrc_decode_workspace_bytes(ct.byref(prm), len(modules), mods, mode, ct.byref(n)), "decode_workspace_bytes")
    if workspace is None or workspace.numel() < n.value:
        workspace = torch.empty(n.value, dtype=torch.uint8, device=dev)
    _check(lib.awsrc_decode_apply(ct.byref(prm), len(modules), mods, _dev_ptr(stream_bytes),
                                  stream_bytes.numel(), int(K), ptrs,
                                  code, mode, _dev_ptr(workspace), workspace.numel(), _stream(stream)),
           "decode_apply")
    outs[0]._awsrc_workspace = workspace
    return outs


def awsrc_decode_apply_inplace_noalloc(prm: Params, modules, stream_bytes: torch.Tensor, K: int,
                                       outs: List[torch.Tensor], stream=None) -> List[torch.Tensor]:
    """In-place decode that allocates nothing on either side of the ABI: `outs`
    must already hold W0; their tiles named by the first K records get W0 + r_hat.
    The library keeps one scratch array per device and uses the current
    device's, so the call runs with the device of `outs` current; the stream
    bytes and every output must live on that device."""
    if not outs:
        raise ValueError("outs must hold one tensor per module")
    dev = outs[0].device
    _require(stream_bytes, "stream_bytes", dtype=torch.uint8, device=dev)
    for i, o in enumerate(outs):
        _require(o, f"outs[{i}]", device=dev)
    _check_outs(modules, outs, modules[0]["W0"].dtype)
    mods = module_array(modules, decoder=True)
    ptrs = (ct.c_void_p * len(outs))(*[_dev_ptr(o) for o in outs])
    with torch.cuda.device(dev):
        _check(lib.awsrc_decode_apply_inplace_noalloc(ct.byref(prm), len(modules), mods, _dev_ptr(stream_bytes),
                                                      stream_bytes.numel(), int(K), ptrs,
                                                      _stream(stream if stream is not None
                                                              else torch.cuda.current_stream(dev))),
               "decode_apply_inplace_noalloc")
    return outs


def awsrc_workspace_status(workspace: torch.Tensor, stream=None) -> int:
    flags = ct.c_uint32()
    _check(lib.awsrc_workspace_status(_dev_ptr(workspace), _stream(stream), ct.byref(flags)), "workspace_status")
    return flags.value


def awsrc_set_timing_events(before: Optional[torch.cuda.Event], after: Optional[torch.cuda.Event]):
    """Record `before`/`after` around the seed-search launches of later encode calls.
    The events must already exist (torch creates them on their first record())."""
    b = before.cuda_event if before is not None else None
    a = after.cuda_event if after is not None else None
    if (before is not None and not b) or (after is not None and not a):
        raise ValueError("record the events once before handing them to the library")
    lib.awsrc_set_timing_events(b, a)


def awsrc_kernel_launches() -> int:
    return int(lib.awsrc_kernel_launches())


def awsrc_set_search_pruning(enabled: bool):
    """For this host thread: False makes later encode calls score every
    candidate (results identical by design; a check of the pruning bound)."""
    lib.awsrc_set_search_pruning(1 if enabled else 0)


def awsrc_set_wait_test(wait_ns: int = 0, stall_chunk: int = -1):
    """For this host thread: the limit of the kernels' bounded waits (0 = 2 s)
    and, for stall_chunk >= 0, the seed chunk from which the C = 64, P = 4 U
    search issues no copies, so that its waits run out (a test of the timeout
    path). awsrc_set_wait_test() restores normal operation."""
    lib.awsrc_set_wait_test(int(wait_ns), int(stall_chunk))


def awsrc_verify_reciprocal(first: int, last: int, stream=None, device="cuda") -> int:
    """Bit patterns in [first, last) where the library's reciprocal differs from
    CUDA's correctly rounded one (synchronises)."""
    bad = torch.zeros(1, dtype=torch.int64, device=device)
    _check(lib.awsrc_verify_reciprocal(first, last, _dev_ptr(bad), _stream(stream)), "verify_reciprocal")
    return int(bad.item())


def candidates_to_numpy(cands: torch.Tensor) -> np.ndarray:
    """Device candidate bytes -> host structured array (gain, seed, scale, code[8])."""
    return cands.cpu().numpy().reshape(-1).view(CANDIDATE_DTYPE)
