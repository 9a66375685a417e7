"""ctypes binding of libe2s.so (include/e2s.h).  Argument marshalling only.

Functions keep the C names and argument order.  Pointer arguments accept a
torch tensor (its data_ptr), a raw integer address, or None (NULL).  Stream
arguments accept a torch.cuda.Stream, a raw cudaStream_t integer, or None
(the legacy default stream).  There is no fallback: importing this module
raises ImportError when the library has not been built.
"""
from __future__ import annotations

import ctypes
import os

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libe2s.so")
if not os.path.exists(_LIB_PATH):
    raise ImportError(f"{_LIB_PATH} is missing: build it with `python -c \"import __graft_entry__ as g; "
                      f"g.build()\"` (nvcc, sm_103a)")
lib = ctypes.CDLL(_LIB_PATH)

# ---- status codes and enums (mirror include/e2s.h)
E2S_OK = 0
E2S_ERR_INVALID_ARG = 1
E2S_ERR_SHAPE = 2
E2S_ERR_ALIGNMENT = 3
E2S_ERR_UNSUPPORTED = 4
E2S_ERR_WORKSPACE = 5
E2S_ERR_CUDA = 6
E2S_ERR_TIMEOUT = 7

E2S_SCORE_EQ1 = 0
E2S_SCORE_CAUSAL_PROB = 1
E2S_NORM_DEFAULT = 0
E2S_NORM_SOFTMAX = 1
E2S_NORM_RENORM = 2

E2S_NO_RELIABILITY = 1 << 0
E2S_NO_LAYER_FUSION = 1 << 1
E2S_NO_CONFLICT = 1 << 2
E2S_NO_NOVELTY = 1 << 3
E2S_VANILLA = 1 << 4
E2S_SIMT_SCORE = 1 << 8

_i32p = ctypes.c_void_p


class e2s_layout(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int32), ("L", ctypes.c_int32), ("H", ctypes.c_int32),
                ("H_kv", ctypes.c_int32), ("d", ctypes.c_int32),
                ("tok_off", _i32p), ("n_sys", _i32p), ("n_vis", _i32p), ("n_text", _i32p),
                ("grid_h", _i32p), ("grid_w", _i32p), ("vis_off", _i32p), ("text_off", _i32p),
                ("max_T", ctypes.c_int32), ("max_vis", ctypes.c_int32), ("max_text", ctypes.c_int32),
                ("sum_T", ctypes.c_int32), ("sum_vis", ctypes.c_int32), ("sum_text", ctypes.c_int32)]


class e2s_params(ctypes.Structure):
    _fields_ = [("lambda_", ctypes.c_float), ("G", ctypes.c_int32), ("score_mode", ctypes.c_int32),
                ("norm_mode", ctypes.c_int32), ("flags", ctypes.c_uint32)]


def params(lam: float = 0.1, G: int = 4, score_mode: int = E2S_SCORE_CAUSAL_PROB,
           norm_mode: int = E2S_NORM_DEFAULT, flags: int = 0) -> e2s_params:
    """Defaults are the paper's: lambda = 0.1, G = 4 (Algorithm 1, Sec. 4.3)."""
    return e2s_params(lam, G, score_mode, norm_mode, flags)


_LP = ctypes.POINTER(e2s_layout)
_PP = ctypes.POINTER(e2s_params)
_vp = ctypes.c_void_p
_i64 = ctypes.c_int64
_i32 = ctypes.c_int32
_sz = ctypes.c_size_t

_SIGS = {
    "e2s_workspace_size": (_sz, [_LP, _PP]),
    "e2s_score": (ctypes.c_int, [_LP, _PP, _vp, _i64, _vp, _i64, _vp, _vp, _sz, _vp]),
    "e2s_score_lse": (ctypes.c_int, [_LP, _PP, _vp, _i64, _vp, _i64, _vp, _vp, _vp, _sz, _vp]),
    "e2s_decide": (ctypes.c_int, [_LP, _PP, _vp, _i64, _vp, _i64, _vp, _vp, _vp, _vp, _vp, _vp,
                                   _vp, _vp, _i32, _vp, _vp, _vp, _sz, _vp]),
    "e2s_decide_lse": (ctypes.c_int, [_LP, _PP, _vp, _i64, _vp, _i64, _vp, _vp, _vp, _vp, _vp,
                                       _vp, _vp, _vp, _vp, _i32, _vp, _vp, _vp, _sz, _vp]),
    "e2s_prune": (ctypes.c_int, [_LP, _PP, _vp, _i64, _vp, _i64, _vp, _vp, _vp, _vp, _vp, _vp,
                                  _vp, _vp, _i32, _vp, _vp, _i32, _vp, _vp, _vp, _vp, _vp, _sz,
                                  _vp]),
    "e2s_prune_lse": (ctypes.c_int, [_LP, _PP, _vp, _i64, _vp, _i64, _vp, _vp, _vp, _vp, _vp,
                                      _vp, _vp, _vp, _vp, _i32, _vp, _vp, _i32, _vp, _vp, _vp,
                                      _vp, _vp, _sz, _vp]),
    "e2s_fuse": (ctypes.c_int, [_LP, _PP, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "e2s_fuse_select": (ctypes.c_int, [_LP, _PP, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _i32,
                                        _vp, _vp, _vp, _sz, _vp]),
    "e2s_fuse_noalloc": (ctypes.c_int, [_LP, _PP, _vp, _vp, _vp, _vp, _vp, _vp, _vp]),
    "e2s_select": (ctypes.c_int, [_LP, _PP, _vp, _vp, _vp, _vp, _i32, _vp, _vp, _vp, _sz, _vp]),
    "e2s_compact": (ctypes.c_int, [_LP, _vp, _vp, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "e2s_read_status": (ctypes.c_int, [_vp, _vp]),
    "e2s_clear_status": (ctypes.c_int, [_vp, _vp]),
    "e2s_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "e2s_attention": (ctypes.c_int, [_LP, _vp, _i64, _vp, _i64, _vp, _i64, _vp, _i64, _vp,
                                      _vp, _vp, _sz, _vp]),
    "e2s_decide_attn": (ctypes.c_int, [_LP, _PP, _vp, _i64, _vp, _i64, _vp, _i64, _vp, _i64,
                                        _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _i32, _vp,
                                        _vp, _vp, _sz, _vp]),
    "e2s_selftest_bounded_wait": (ctypes.c_int, [_i32, _i64, _vp, _vp]),
    "e2s_version": (ctypes.c_int32, []),
}
for _name, (_res, _args) in _SIGS.items():
    _f = getattr(lib, _name)
    _f.restype = _res
    _f.argtypes = _args

EXPORTED = tuple(_SIGS)


class E2SError(RuntimeError):
    def __init__(self, status: int, where: str = ""):
        super().__init__(f"{where}: {e2s_status_string(status)} ({status})")
        self.status = status


def _ptr(x) -> int:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _stream(s) -> int:
    if s is None:
        return None
    if isinstance(s, int):
        return s
    return s.cuda_stream


def _ref(x):
    return None if x is None else ctypes.byref(x)


def e2s_workspace_size(layout: e2s_layout, params_: e2s_params) -> int:
    return int(lib.e2s_workspace_size(_ref(layout), _ref(params_)))


def e2s_score(layout, params_, q_text, q_row_stride, k, k_row_stride, a_out, ws, ws_bytes,
              stream=None) -> int:
    return lib.e2s_score(_ref(layout), _ref(params_), _ptr(q_text), q_row_stride, _ptr(k),
                         k_row_stride, _ptr(a_out), _ptr(ws), ws_bytes, _stream(stream))


def e2s_score_lse(layout, params_, q_text, q_row_stride, k, k_row_stride, lse_text, a_out, ws,
                  ws_bytes, stream=None) -> int:
    return lib.e2s_score_lse(_ref(layout), _ref(params_), _ptr(q_text), q_row_stride, _ptr(k),
                             k_row_stride, _ptr(lse_text), _ptr(a_out), _ptr(ws), ws_bytes,
                             _stream(stream))


def e2s_decide_lse(layout, params_, q_text, q_row_stride, k, k_row_stride, lse_text, cand, prior,
                   a_out, mass_out, fused_out, q_out, keep_count, keep_off, sum_keep, keep_idx,
                   q_tilde_out, ws, ws_bytes, stream=None) -> int:
    return lib.e2s_decide_lse(_ref(layout), _ref(params_), _ptr(q_text), q_row_stride, _ptr(k),
                              k_row_stride, _ptr(lse_text), _ptr(cand), _ptr(prior), _ptr(a_out),
                              _ptr(mass_out), _ptr(fused_out), _ptr(q_out), _ptr(keep_count),
                              _ptr(keep_off), sum_keep, _ptr(keep_idx), _ptr(q_tilde_out),
                              _ptr(ws), ws_bytes, _stream(stream))


def e2s_decide(layout, params_, q_text, q_row_stride, k, k_row_stride, cand, prior, a_out,
               mass_out, fused_out, q_out, keep_count, keep_off, sum_keep, keep_idx, q_tilde_out,
               ws, ws_bytes, stream=None) -> int:
    return lib.e2s_decide(_ref(layout), _ref(params_), _ptr(q_text), q_row_stride, _ptr(k),
                          k_row_stride, _ptr(cand), _ptr(prior), _ptr(a_out), _ptr(mass_out),
                          _ptr(fused_out), _ptr(q_out), _ptr(keep_count), _ptr(keep_off),
                          sum_keep, _ptr(keep_idx), _ptr(q_tilde_out), _ptr(ws), ws_bytes,
                          _stream(stream))


def _addr_arrays(src, dst, row_bytes, n):
    src_a = (ctypes.c_void_p * max(n, 1))(*[_ptr(x) for x in src])
    dst_a = (ctypes.c_void_p * max(n, 1))(*[_ptr(x) for x in dst])
    rb_a = (ctypes.c_int64 * max(n, 1))(*[int(x) for x in row_bytes])
    return (ctypes.cast(src_a, ctypes.c_void_p), ctypes.cast(dst_a, ctypes.c_void_p),
            ctypes.cast(rb_a, ctypes.c_void_p), (src_a, dst_a, rb_a))


def e2s_prune_lse(layout, params_, q_text, q_row_stride, k, k_row_stride, lse_text, cand, prior,
                  a_out, mass_out, fused_out, q_out, keep_count, keep_off, sum_keep, keep_idx,
                  q_tilde_out, n_tensors, src, dst, row_bytes, pos_ids_out, ws, ws_bytes,
                  stream=None) -> int:
    """src/dst: sequences of tensors or addresses; row_bytes: sequence of ints."""
    n = int(n_tensors)
    s_p, d_p, r_p, _keep = _addr_arrays(src, dst, row_bytes, n)
    return lib.e2s_prune_lse(_ref(layout), _ref(params_), _ptr(q_text), q_row_stride, _ptr(k),
                             k_row_stride, _ptr(lse_text), _ptr(cand), _ptr(prior), _ptr(a_out),
                             _ptr(mass_out), _ptr(fused_out), _ptr(q_out), _ptr(keep_count),
                             _ptr(keep_off), sum_keep, _ptr(keep_idx), _ptr(q_tilde_out), n,
                             s_p, d_p, r_p, _ptr(pos_ids_out), _ptr(ws), ws_bytes,
                             _stream(stream))


def e2s_prune(layout, params_, q_text, q_row_stride, k, k_row_stride, cand, prior, a_out,
              mass_out, fused_out, q_out, keep_count, keep_off, sum_keep, keep_idx, q_tilde_out,
              n_tensors, src, dst, row_bytes, pos_ids_out, ws, ws_bytes, stream=None) -> int:
    """src/dst: sequences of tensors or addresses; row_bytes: sequence of ints."""
    n = int(n_tensors)
    s_p, d_p, r_p, _keep = _addr_arrays(src, dst, row_bytes, n)
    return lib.e2s_prune(_ref(layout), _ref(params_), _ptr(q_text), q_row_stride, _ptr(k),
                         k_row_stride, _ptr(cand), _ptr(prior), _ptr(a_out), _ptr(mass_out),
                         _ptr(fused_out), _ptr(q_out), _ptr(keep_count), _ptr(keep_off),
                         sum_keep, _ptr(keep_idx), _ptr(q_tilde_out), n, s_p, d_p, r_p,
                         _ptr(pos_ids_out), _ptr(ws), ws_bytes, _stream(stream))


def e2s_fuse(layout, params_, a, cand, prior, mass_out, fused_out, q_out, ws, ws_bytes,
             stream=None) -> int:
    return lib.e2s_fuse(_ref(layout), _ref(params_), _ptr(a), _ptr(cand), _ptr(prior),
                        _ptr(mass_out), _ptr(fused_out), _ptr(q_out), _ptr(ws), ws_bytes,
                        _stream(stream))


def e2s_fuse_select(layout, params_, a, cand, prior, mass_out, fused_out, q_out, keep_count,
                    keep_off, sum_keep, keep_idx, q_tilde_out, ws, ws_bytes, stream=None) -> int:
    return lib.e2s_fuse_select(_ref(layout), _ref(params_), _ptr(a), _ptr(cand), _ptr(prior),
                               _ptr(mass_out), _ptr(fused_out), _ptr(q_out), _ptr(keep_count),
                               _ptr(keep_off), sum_keep, _ptr(keep_idx), _ptr(q_tilde_out),
                               _ptr(ws), ws_bytes, _stream(stream))


def e2s_attention(layout, q, q_row_stride, k, k_row_stride, v, v_row_stride, o_out,
                  o_row_stride, lse_out, a_out, ws, ws_bytes, stream=None) -> int:
    return lib.e2s_attention(_ref(layout), _ptr(q), q_row_stride, _ptr(k), k_row_stride, _ptr(v),
                             v_row_stride, _ptr(o_out), o_row_stride, _ptr(lse_out), _ptr(a_out),
                             _ptr(ws), ws_bytes, _stream(stream))


def e2s_decide_attn(layout, params_, q, q_row_stride, k, k_row_stride, v, v_row_stride, o_out,
                    o_row_stride, lse_out, cand, prior, a_out, mass_out, fused_out, q_out,
                    keep_count, keep_off, sum_keep, keep_idx, q_tilde_out, ws, ws_bytes,
                    stream=None) -> int:
    return lib.e2s_decide_attn(_ref(layout), _ref(params_), _ptr(q), q_row_stride, _ptr(k),
                               k_row_stride, _ptr(v), v_row_stride, _ptr(o_out), o_row_stride,
                               _ptr(lse_out), _ptr(cand), _ptr(prior), _ptr(a_out),
                               _ptr(mass_out), _ptr(fused_out), _ptr(q_out), _ptr(keep_count),
                               _ptr(keep_off), sum_keep, _ptr(keep_idx), _ptr(q_tilde_out),
                               _ptr(ws), ws_bytes, _stream(stream))


def e2s_selftest_bounded_wait(complete: int, limit_ns: int, ws, stream=None) -> int:
    return lib.e2s_selftest_bounded_wait(int(complete), int(limit_ns), _ptr(ws), _stream(stream))


def e2s_fuse_noalloc(layout, params_, a, cand, prior, mass_out, fused_out, q_out,
                     stream=None) -> int:
    """e2s_fuse with its scratch in a static device array: no workspace, no allocation."""
    return lib.e2s_fuse_noalloc(_ref(layout), _ref(params_), _ptr(a), _ptr(cand), _ptr(prior),
                                _ptr(mass_out), _ptr(fused_out), _ptr(q_out), _stream(stream))


def e2s_select(layout, params_, q, cand, keep_count, keep_off, sum_keep, keep_idx, q_tilde_out,
               ws, ws_bytes, stream=None) -> int:
    return lib.e2s_select(_ref(layout), _ref(params_), _ptr(q), _ptr(cand), _ptr(keep_count),
                          _ptr(keep_off), sum_keep, _ptr(keep_idx), _ptr(q_tilde_out), _ptr(ws),
                          ws_bytes, _stream(stream))


def e2s_compact(layout, keep_idx, keep_off, sum_keep, n_tensors, src, dst, row_bytes, pos_ids_out,
                ws, ws_bytes, stream=None) -> int:
    """src/dst: sequences of tensors or addresses; row_bytes: sequence of ints."""
    n = int(n_tensors)
    s_p, d_p, r_p, _keep = _addr_arrays(src, dst, row_bytes, n)
    return lib.e2s_compact(_ref(layout), _ptr(keep_idx), _ptr(keep_off), sum_keep, n, s_p, d_p,
                           r_p, _ptr(pos_ids_out), _ptr(ws), ws_bytes, _stream(stream))


def e2s_read_status(ws, stream=None) -> int:
    return lib.e2s_read_status(_ptr(ws), _stream(stream))


def e2s_clear_status(ws, stream=None) -> int:
    return lib.e2s_clear_status(_ptr(ws), _stream(stream))


def e2s_status_string(status: int) -> str:
    return lib.e2s_status_string(int(status)).decode()


def e2s_version() -> int:
    return int(lib.e2s_version())


def check(status: int, where: str = "e2s") -> None:
    if status != E2S_OK:
        raise E2SError(status, where)
