"""ctypes binding of include/selkv.h (argument marshalling only)."""
from __future__ import annotations

import ctypes
import os
import re
from typing import Optional

_PKG = os.path.dirname(os.path.abspath(__file__))
_HEADER = os.path.join(os.path.dirname(_PKG), "include", "selkv.h")

SELKV_OK, SELKV_ERR_INVALID_ARG, SELKV_ERR_UNSUPPORTED, SELKV_ERR_WORKSPACE = 0, 1, 2, 3
SELKV_ERR_CUDA, SELKV_ERR_DEVICE = 4, 5
SELKV_BF16, SELKV_FP32 = 0, 1
SELKV_GATE_COSINE, SELKV_GATE_OPEN, SELKV_GATE_CLOSED = 0, 1, 2
SELKV_EMPTY_EXPAND, SELKV_EMPTY_DROP = 0, 1
SELKV_SELECT_SHARED, SELKV_SELECT_PER_HEAD = 0, 1
SELKV_ROPE_OFF, SELKV_ROPE_HALF, SELKV_ROPE_INTERLEAVED = 0, 1, 2
SELKV_BIAS_RATIO, SELKV_BIAS_COUNT = 0, 1
SELKV_ROUTE_BUCKET, SELKV_ROUTE_COSINE = 0, 1
SELKV_SCORE_ROWSTATS, SELKV_SCORE_COLSUMS, SELKV_SCORE_ALL = 1, 2, 3
SELKV_DEVERR_CAPACITY, SELKV_DEVERR_TIMEOUT, SELKV_DEVERR_LENGTH, SELKV_DEVERR_COUNT = 1, 2, 4, 8
SELKV_MAX_BATCH = 1024
SELKV_STATIC_SCRATCH_BYTES = 4 << 20

c_i32, c_u32, c_u64, c_sz, c_vp, c_f32, c_f64 = (ctypes.c_int32, ctypes.c_uint32, ctypes.c_uint64,
                                                 ctypes.c_size_t, ctypes.c_void_p, ctypes.c_float,
                                                 ctypes.c_double)


class SelKVError(RuntimeError):
    def __init__(self, status: int, what: str = ""):
        self.status = status
        detail = ""
        if status == SELKV_ERR_CUDA:
            code, name = selkv_last_cuda_error()
            detail = "; %s (%d)" % (name, code)
        super().__init__("%s: %s (status %d%s)" % (what or "selkv", selkv_status_string(status), status, detail))


class selkv_shape(ctypes.Structure):
    _fields_ = [("dtype", c_i32), ("batch", c_i32), ("num_q_heads", c_i32), ("num_kv_heads", c_i32),
                ("head_dim", c_i32), ("obs_window", c_i32), ("n_cap", c_i32), ("m_cap", c_i32)]


class selkv_params(ctypes.Structure):
    _fields_ = [("alpha", c_f32), ("pool_kernel", c_i32), ("bucket", c_i32), ("recent", c_i32),
                ("gate_mode", c_i32), ("empty_bucket", c_i32), ("select_mode", c_i32),
                ("rope", c_i32), ("rope_theta", c_f32), ("bias_mode", c_i32),
                ("routing", c_i32)]

    @classmethod
    def defaults(cls, **kw) -> "selkv_params":
        """The paper's configuration (Sec. 4.1 / App. F): alpha 0.5, K 5, B 32, m_r 16."""
        p = dict(alpha=0.5, pool_kernel=5, bucket=32, recent=16, gate_mode=SELKV_GATE_COSINE,
                 empty_bucket=SELKV_EMPTY_EXPAND, select_mode=SELKV_SELECT_SHARED,
                 rope=SELKV_ROPE_OFF, rope_theta=10000.0, bias_mode=SELKV_BIAS_RATIO,
                 routing=SELKV_ROUTE_BUCKET)
        p.update(kw)
        return cls(**p)


class selkv_compress_debug(ctypes.Structure):
    _fields_ = [("attn", c_vp), ("score", c_vp), ("topk", c_vp), ("kept_idx", c_vp),
                ("target", c_vp), ("gate", c_vp), ("decision", c_vp), ("ratio", c_vp)]


_LIB: Optional[ctypes.CDLL] = None


def library_path() -> str:
    return os.path.join(_PKG, "_lib", "libselkv.so")


def library() -> ctypes.CDLL:
    """Load libselkv.so (once).  Raises if it has not been built."""
    global _LIB
    if _LIB is not None:
        return _LIB
    path = library_path()
    if not os.path.exists(path):
        raise RuntimeError("SelKV CUDA library not built (%s missing): run "
                           "`python -c 'import __graft_entry__ as g; g.build()'`" % path)
    lib = ctypes.CDLL(path)
    sig = {
        "selkv_status_string": (ctypes.c_char_p, [c_i32]),
        "selkv_last_cuda_error": (c_i32, [ctypes.POINTER(ctypes.c_char_p)]),
        "selkv_kernel_launches": (c_u64, []),
        "selkv_workspace_init": (c_i32, [c_vp, c_sz, c_vp]),
        "selkv_workspace_error": (c_i32, [c_vp, c_vp, ctypes.POINTER(c_u32)]),
        "selkv_compress_workspace_size": (c_sz, [ctypes.POINTER(selkv_shape)]),
        "selkv_compress": (c_i32, [ctypes.POINTER(selkv_shape), ctypes.POINTER(c_i32), c_f64,
                                   ctypes.POINTER(selkv_params), c_vp, c_vp, c_vp, c_vp, c_vp, c_vp,
                                   c_vp, ctypes.POINTER(selkv_compress_debug), c_vp, c_sz, c_vp]),
        "selkv_score_workspace_size": (c_sz, [ctypes.POINTER(selkv_shape)]),
        "selkv_score": (c_i32, [ctypes.POINTER(selkv_shape), ctypes.POINTER(c_i32), c_vp, c_vp, c_vp, c_i32,
                                c_vp, c_sz, c_vp]),
        "selkv_layer_average_workspace_size": (c_sz, [ctypes.POINTER(selkv_shape)]),
        "selkv_layer_average_bias": (c_i32, [ctypes.POINTER(selkv_shape), ctypes.POINTER(selkv_params), c_i32,
                                             ctypes.POINTER(c_vp), ctypes.POINTER(c_vp), c_vp, c_vp, c_sz,
                                             c_vp]),
        "selkv_decode_workspace_size": (c_sz, [ctypes.POINTER(selkv_shape)]),
        "selkv_decode_attn": (c_i32, [ctypes.POINTER(selkv_shape), c_vp, c_vp, c_vp, c_vp, c_vp,
                                      c_vp, c_vp, c_vp, c_vp, c_sz, c_vp]),
        "selkv_decode_attn_static": (c_i32, [ctypes.POINTER(selkv_shape), c_vp, c_vp, c_vp, c_vp,
                                             c_vp, c_vp, c_vp, c_vp, c_vp, c_vp]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _LIB = lib
    return lib


def exported_symbols() -> list:
    """Names of the functions include/selkv.h declares."""
    text = open(_HEADER).read()
    return sorted(set(re.findall(r"^SELKV_API\s+[\w\s\*]+?\b(selkv_\w+)\s*\(", text, re.M)))


def _ptr(x) -> Optional[int]:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def check(status: int, what: str = "") -> None:
    if status != SELKV_OK:
        raise SelKVError(status, what)


def selkv_status_string(status: int) -> str:
    try:
        return library().selkv_status_string(status).decode()
    except RuntimeError:
        return "status %d" % status


def selkv_last_cuda_error():
    """(code, name) of the CUDA error behind the last SELKV_ERR_CUDA on this thread."""
    try:
        name = ctypes.c_char_p()
        code = int(library().selkv_last_cuda_error(ctypes.byref(name)))
        return code, (name.value or b"").decode()
    except RuntimeError:
        return -1, "unknown"


def selkv_kernel_launches() -> int:
    return int(library().selkv_kernel_launches())


def selkv_workspace_init(workspace, workspace_bytes: int, stream=None) -> int:
    return library().selkv_workspace_init(_ptr(workspace), workspace_bytes, _stream(stream))


def selkv_workspace_error(workspace, stream=None):
    """Returns (status, flags)."""
    f = c_u32(0)
    st = library().selkv_workspace_error(_ptr(workspace), _stream(stream), ctypes.byref(f))
    return st, int(f.value)


def selkv_compress_workspace_size(shape: selkv_shape) -> int:
    return int(library().selkv_compress_workspace_size(ctypes.byref(shape)))


def selkv_score_workspace_size(shape: selkv_shape) -> int:
    return int(library().selkv_score_workspace_size(ctypes.byref(shape)))


def selkv_score(shape: selkv_shape, n_len, K, Q_obs, attn, passes: int, workspace, workspace_bytes: int,
                stream=None) -> int:
    """See include/selkv.h.  n_len: host sequence of B ints."""
    n_arr = (c_i32 * shape.batch)(*[int(x) for x in n_len])
    return library().selkv_score(ctypes.byref(shape), n_arr, _ptr(K), _ptr(Q_obs), _ptr(attn), int(passes),
                                 _ptr(workspace), int(workspace_bytes), _stream(stream))


def selkv_layer_average_workspace_size(shape: selkv_shape) -> int:
    return library().selkv_layer_average_workspace_size(ctypes.byref(shape))


def selkv_layer_average_bias(shape: selkv_shape, params: selkv_params, kept_idx, bias, lengths,
                             workspace, workspace_bytes: int, stream=None) -> int:
    """kept_idx, bias: sequences of per-layer tensors (or device addresses)."""
    L = len(kept_idx)
    kept_arr = (c_vp * L)(*[_ptr(k) for k in kept_idx])
    bias_arr = (c_vp * L)(*[_ptr(b) for b in bias])
    return library().selkv_layer_average_bias(ctypes.byref(shape), ctypes.byref(params), L, kept_arr, bias_arr,
                                              _ptr(lengths), _ptr(workspace), workspace_bytes, _stream(stream))


def selkv_decode_workspace_size(shape: selkv_shape) -> int:
    return int(library().selkv_decode_workspace_size(ctypes.byref(shape)))


def selkv_compress(shape: selkv_shape, n_len, rho: float, params: selkv_params, K, V, Q_obs,
                   K_c, V_c, bias, lengths, debug: Optional[dict] = None, workspace=None,
                   workspace_bytes: int = 0, stream=None) -> int:
    """See include/selkv.h.  n_len: host sequence of B ints.  debug: optional dict with any of
    the selkv_compress_debug fields mapped to device tensors."""
    n_arr = (c_i32 * shape.batch)(*[int(x) for x in n_len])
    dbg = None
    if debug:
        dbg = selkv_compress_debug(**{k: _ptr(v) for k, v in debug.items()})
    return library().selkv_compress(ctypes.byref(shape), n_arr, float(rho), ctypes.byref(params),
                                    _ptr(K), _ptr(V), _ptr(Q_obs), _ptr(K_c), _ptr(V_c), _ptr(bias),
                                    _ptr(lengths), ctypes.byref(dbg) if dbg is not None else None,
                                    _ptr(workspace), int(workspace_bytes), _stream(stream))


def selkv_decode_attn(shape: selkv_shape, q, K_c, V_c, bias, lengths, k_new, v_new, out,
                      workspace, workspace_bytes: int, stream=None) -> int:
    """See include/selkv.h."""
    return library().selkv_decode_attn(ctypes.byref(shape), _ptr(q), _ptr(K_c), _ptr(V_c), _ptr(bias),
                                       _ptr(lengths), _ptr(k_new), _ptr(v_new), _ptr(out),
                                       _ptr(workspace), int(workspace_bytes), _stream(stream))


def selkv_decode_attn_static(shape: selkv_shape, q, K_c, V_c, bias, lengths, k_new, v_new, out,
                             flags_out=None, stream=None) -> int:
    """See include/selkv.h: the decode for callers that cannot allocate (no workspace)."""
    return library().selkv_decode_attn_static(ctypes.byref(shape), _ptr(q), _ptr(K_c), _ptr(V_c),
                                              _ptr(bias), _ptr(lengths), _ptr(k_new), _ptr(v_new),
                                              _ptr(out), _ptr(flags_out), _stream(stream))
