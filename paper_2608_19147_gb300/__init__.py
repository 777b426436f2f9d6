"""Python binding of libshard (include/shard.h, include/shard_debug.h,
include/head.h).

Argument marshalling only: every function forwards to the C ABI function of
the same name, which runs the work in the library's CUDA kernels.  Device
pointers are passed as integers (e.g. ``tensor.data_ptr()``); host buffers as
numpy arrays.  Importing the package does not need a GPU; calling into the
library does, and there is no fallback: if libshard.so is missing the calls
raise.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libshard.so")

SHARD_OK, SHARD_EINVAL, SHARD_ECAPACITY, SHARD_ENOMEM, SHARD_ECUDA, SHARD_EUNSUPPORTED = 0, -1, -2, -3, -4, -5
SHARD_MAX_TOKENS = 16
SHARD_MAX_REQUESTS = 16
OP_QKV, OP_O, OP_GU, OP_DOWN = 0, 1, 2, 3

# Every symbol include/shard.h and include/shard_debug.h declare.
EXPORTS = ("shard_create", "shard_destroy", "kv_state_alloc", "kv_state_free", "kv_state_reset", "kv_state_load",
           "kv_state_read", "kv_state_length", "kv_trim", "kv_state_export", "kv_state_import", "shard_step", "shard_step_packed", "shard_prefill", "shard_step_host", "shard_sync_status",
           "shard_last_error", "shard_debug_op_info", "shard_debug_unpack", "shard_debug_gemv", "shard_debug_gemm",
           "shard_debug_phase_times", "shard_debug_set_wait", "shard_gemv_noalloc", "head_create", "head_destroy", "head_top1",
           "head_top1_host", "head_debug_logits")
# per layer, between the ends of grid-barrier waits: attention (with the next
# layer's RMSNorm + q|k|v projection in front of it after the first layer), o,
# RMSNorm + gate|up, down; before them the prologue with the first RMSNorm and
# q|k|v projection
PHASES = ("attention", "o", "gate_up", "down")


class ShardError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__("libshard error %d: %s" % (code, msg))
        self.code = code


class shard_config(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("hidden", ctypes.c_int32), ("n_heads", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32), ("ffn", ctypes.c_int32),
                ("group", ctypes.c_int32), ("vocab", ctypes.c_int32), ("max_position", ctypes.c_int32),
                ("reserved", ctypes.c_int32), ("rms_eps", ctypes.c_double), ("rope_theta", ctypes.c_double)]


class shard_matrix_host(ctypes.Structure):
    _fields_ = [("codes", ctypes.c_void_p), ("scales", ctypes.c_void_p), ("zeros", ctypes.c_void_p)]


class shard_layer_host(ctypes.Structure):
    _fields_ = [("w", shard_matrix_host * 7), ("attn_norm", ctypes.c_void_p), ("ffn_norm", ctypes.c_void_p)]


class shard_weights_host(ctypes.Structure):
    _fields_ = [("layers", ctypes.POINTER(shard_layer_host)), ("embedding", ctypes.c_void_p)]


class head_config(ctypes.Structure):
    _fields_ = [("hidden", ctypes.c_int32), ("vocab", ctypes.c_int32), ("group", ctypes.c_int32),
                ("reserved", ctypes.c_int32), ("rms_eps", ctypes.c_double)]


class head_weights_host(ctypes.Structure):
    _fields_ = [("lm_head", shard_matrix_host), ("norm", ctypes.c_void_p)]


_lib = None


def load_library(path: str = LIB_PATH):
    """Loads libshard.so; raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise ImportError("libshard.so not found at %s: build it with __graft_entry__.build() "
                          "or python paper_2608_19147_gb300/build.py" % path)
    lib = ctypes.CDLL(path)
    vp, ip, i32p = ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p
    sig = {
        "shard_create": ([ctypes.POINTER(shard_config), ctypes.POINTER(shard_weights_host), ctypes.POINTER(vp)], ip),
        "shard_destroy": ([vp], ip),
        "kv_state_alloc": ([vp, ip, ip, ctypes.POINTER(vp)], ip),
        "kv_state_free": ([vp], ip),
        "kv_state_reset": ([vp, ip], ip),
        "kv_state_load": ([vp, ip, ip, vp, vp, ip], ip),
        "kv_state_read": ([vp, ip, ip, ip, ip, vp, vp], ip),
        "kv_state_length": ([vp, ip, ctypes.POINTER(ctypes.c_int)], ip),
        "kv_trim": ([vp, ip, vp, ip], ip),
        "kv_state_export": ([vp, ip, vp, ip, vp, vp, ctypes.POINTER(ctypes.c_int)], ip),
        "kv_state_import": ([vp, ip, vp, vp, ip], ip),
        "shard_step": ([vp, vp, vp, vp, i32p, ip, vp, vp, ip, vp, vp, vp], ip),
        "shard_step_host": ([vp, vp, vp, vp, i32p, ip, vp, vp, ip, vp, vp, vp], ip),
        "shard_step_packed": ([vp, vp, vp, vp, ip, vp, vp, ip, vp, vp], ip),
        "shard_prefill": ([vp, vp, ip, vp, vp, ip, vp, vp, ip, vp, vp], ip),
        "shard_sync_status": ([vp, vp], ip),
        "shard_last_error": ([], ctypes.c_char_p),
        "shard_debug_op_info": ([vp, ip, ip, ctypes.POINTER(ctypes.c_int), ctypes.POINTER(ctypes.c_int),
                                 ctypes.POINTER(ctypes.c_longlong)], ip),
        "shard_debug_unpack": ([vp, ip, ip, vp, ip], ip),
        "shard_debug_gemv": ([vp, ip, ip, vp, ip, vp, ip, vp], ip),
        "shard_gemv_noalloc": ([vp, ip, ip, vp, ip, vp, ip, vp], ip),
        "shard_debug_phase_times": ([vp, ctypes.POINTER(ctypes.c_double), ip], ip),
        "shard_debug_gemm": ([vp, ip, ip, vp, ip, ip, vp, ip, vp], ip),
        "shard_debug_set_wait": ([vp, ctypes.c_uint, ip], ip),
        "head_create": ([ctypes.POINTER(head_config), ctypes.POINTER(head_weights_host), ctypes.POINTER(vp)], ip),
        "head_destroy": ([vp], ip),
        "head_top1": ([vp, vp, ip, vp, vp, vp], ip),
        "head_top1_host": ([vp, vp, ip, vp, vp, vp], ip),
        "head_debug_logits": ([vp, vp, ip, vp, ip, vp], ip),
    }
    for name, (args, res) in sig.items():
        f = getattr(lib, name)
        f.argtypes = args
        f.restype = res
    _lib = lib
    return lib


def _check(rc: int) -> int:
    if rc != SHARD_OK:
        raise ShardError(rc, shard_last_error())
    return rc


def _np(a: Optional[np.ndarray], dtype=None):
    if a is None:
        return None
    if dtype is not None:
        assert a.dtype == dtype, (a.dtype, dtype)
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data


def shard_last_error() -> str:
    return load_library().shard_last_error().decode()


def make_config(shape) -> shard_config:
    """shard_config from any object with the shard shape's attribute names."""
    return shard_config(shape.n_layers, shape.hidden, shape.n_heads, shape.n_kv_heads, shape.head_dim, shape.ffn,
                        shape.group, shape.vocab, shape.max_position, 0, float(shape.rms_eps),
                        float(shape.rope_theta))


def shard_create(cfg: shard_config, layers: Sequence, embedding: Optional[np.ndarray]) -> int:
    """layers: per layer (matrices[7] with .codes/.scales/.zeros arrays, attn_norm, ffn_norm)."""
    lib = load_library()
    arr = (shard_layer_host * len(layers))()
    for i, lw in enumerate(layers):
        for j, m in enumerate(lw.matrices):
            arr[i].w[j] = shard_matrix_host(_np(m.codes, np.uint8), _np(m.scales, np.uint16), _np(m.zeros, np.uint8))
        arr[i].attn_norm = _np(lw.attn_norm, np.uint16)
        arr[i].ffn_norm = _np(lw.ffn_norm, np.uint16)
    w = shard_weights_host(arr, _np(embedding, np.uint16))
    out = ctypes.c_void_p()
    _check(lib.shard_create(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(out)))
    return out.value


def shard_destroy(shard: int) -> None:
    _check(load_library().shard_destroy(shard))


def kv_state_alloc(shard: int, n_rows: int, capacity: int) -> int:
    out = ctypes.c_void_p()
    _check(load_library().kv_state_alloc(shard, n_rows, capacity, ctypes.byref(out)))
    return out.value


def kv_state_free(state: int) -> None:
    _check(load_library().kv_state_free(state))


def kv_state_reset(state: int, row: int) -> None:
    _check(load_library().kv_state_reset(state, row))


def kv_state_load(state: int, row: int, layer: int, k: np.ndarray, v: np.ndarray) -> None:
    k = np.ascontiguousarray(k, dtype=np.uint16)
    v = np.ascontiguousarray(v, dtype=np.uint16)
    _check(load_library().kv_state_load(state, row, layer, _np(k), _np(v), k.shape[0]))


def kv_state_read(state: int, row: int, layer: int, start: int, length: int, n_kv_heads: int, head_dim: int):
    k = np.empty((length, n_kv_heads, head_dim), dtype=np.uint16)
    v = np.empty_like(k)
    _check(load_library().kv_state_read(state, row, layer, start, length, _np(k), _np(v)))
    return k, v


def kv_state_length(state: int, row: int) -> int:
    n = ctypes.c_int()
    _check(load_library().kv_state_length(state, row, ctypes.byref(n)))
    return n.value


def kv_trim(state: int, row: int, keep: np.ndarray) -> None:
    keep = np.ascontiguousarray(keep, dtype=np.uint8)
    _check(load_library().kv_trim(state, row, _np(keep), keep.size))


def kv_state_export(state: int, row: int, length: int, n_layers: int, n_kv_heads: int, head_dim: int,
                    keep: Optional[np.ndarray] = None):
    """Compacted copy of the row's entries with keep != 0 (all when None):
    (k, v), each [n_layers][n_kept][Hkv][d] fp16 bits."""
    per = n_kv_heads * head_dim
    k = np.empty(n_layers * max(length, 1) * per, dtype=np.uint16)
    v = np.empty_like(k)
    kp = None if keep is None else np.ascontiguousarray(keep, dtype=np.uint8)
    n = ctypes.c_int()
    _check(load_library().kv_state_export(state, row, _np(kp), length, _np(k), _np(v), ctypes.byref(n)))
    shape = (n_layers, n.value, n_kv_heads, head_dim)  # packed: [n_layers][n_kept][Hkv][d]
    return k[:n_layers * n.value * per].reshape(shape).copy(), v[:n_layers * n.value * per].reshape(shape).copy()


def kv_state_import(state: int, row: int, k: np.ndarray, v: np.ndarray) -> None:
    """k, v: [n_layers][len][Hkv][d] fp16 bits (as kv_state_export returns)."""
    k = np.ascontiguousarray(k, dtype=np.uint16)
    v = np.ascontiguousarray(v, dtype=np.uint16)
    _check(load_library().kv_state_import(state, row, _np(k), _np(v), k.shape[1]))


def shard_step(shard: int, state: int, hidden_in: Optional[int], token_ids: Optional[int], n_new: Sequence[int],
               position_ids: int, attention_mask: int, mask_stride: int, beam_idx: Optional[int], hidden_out: int,
               stream: int = 0, check: bool = True) -> int:
    """Device pointers as ints (0/None for absent ones); n_new is host data."""
    n = np.ascontiguousarray(n_new, dtype=np.int32)
    rc = load_library().shard_step(shard, state, hidden_in or None, token_ids or None, _np(n), len(n), position_ids,
                                   attention_mask, mask_stride, beam_idx or None, hidden_out, stream or None)
    return _check(rc) if check else rc


def shard_step_packed(shard: int, state: int, hidden_in: Optional[int], token_ids: Optional[int], S: int,
                      position_ids: int, mask2d: int, mask_stride: int, hidden_out: int, stream: int = 0,
                      check: bool = True) -> int:
    """Packed step (Section 8.6): device pointers as ints; mask2d [S][mask_stride]."""
    rc = load_library().shard_step_packed(shard, state, hidden_in or None, token_ids or None, S, position_ids, mask2d,
                                          mask_stride, hidden_out, stream or None)
    return _check(rc) if check else rc


def shard_prefill(shard: int, state: int, row: int, hidden_in: Optional[int], token_ids: Optional[int], S: int,
                  position_ids: int, attention_mask: int, mask_len: int, hidden_out: int, stream: int = 0,
                  check: bool = True) -> int:
    """Prefill of one row (device pointers as ints)."""
    rc = load_library().shard_prefill(shard, state, row, hidden_in or None, token_ids or None, S, position_ids,
                                      attention_mask, mask_len, hidden_out, stream or None)
    return _check(rc) if check else rc


def shard_step_host(shard: int, state: int, hidden_in: Optional[np.ndarray], token_ids: Optional[np.ndarray],
                    n_new: Sequence[int], position_ids: np.ndarray, attention_mask: np.ndarray,
                    beam_idx: Optional[np.ndarray], hidden_out: np.ndarray, stream: int = 0,
                    check: bool = True) -> int:
    n = np.ascontiguousarray(n_new, dtype=np.int32)
    mask = np.ascontiguousarray(attention_mask, dtype=np.uint8)
    stride = mask.shape[-1]
    rc = load_library().shard_step_host(
        shard, state, _np(hidden_in, np.uint16), _np(token_ids, np.int32), _np(n), len(n),
        _np(np.ascontiguousarray(position_ids, dtype=np.int32)), _np(mask), stride,
        _np(beam_idx, np.int32), _np(hidden_out, np.uint16), stream or None)
    return _check(rc) if check else rc


def shard_sync_status(shard: int, stream: int = 0, check: bool = True) -> int:
    rc = load_library().shard_sync_status(shard, stream or None)
    return _check(rc) if check else rc


def shard_debug_op_info(shard: int, layer: int, op: int):
    rows, K, nbytes = ctypes.c_int(), ctypes.c_int(), ctypes.c_longlong()
    _check(load_library().shard_debug_op_info(shard, layer, op, ctypes.byref(rows), ctypes.byref(K),
                                              ctypes.byref(nbytes)))
    return rows.value, K.value, nbytes.value


def shard_debug_unpack(shard: int, layer: int, op: int, out: int, ld: int) -> None:
    _check(load_library().shard_debug_unpack(shard, layer, op, out, ld))


def shard_debug_gemv(shard: int, layer: int, op: int, x: int, M: int, y: int, y_ld: int, stream: int = 0) -> None:
    _check(load_library().shard_debug_gemv(shard, layer, op, x, M, y, y_ld, stream or None))


def shard_debug_gemm(shard: int, layer: int, op: int, x: int, x_ld: int, S: int, y: int, y_ld: int,
                     stream: int = 0) -> None:
    """Many-token tensor-core projection (device pointers as ints; x padded to x_ld)."""
    _check(load_library().shard_debug_gemm(shard, layer, op, x, x_ld, S, y, y_ld, stream or None))


def shard_debug_phase_times(shard: int, n_layers: int):
    """Durations (microseconds) of the last step's phases: the prologue (with
    the first RMSNorm and q|k|v projection), then per layer the phases named
    in PHASES."""
    n = len(PHASES) * n_layers + 1
    buf = (ctypes.c_double * n)()
    k = load_library().shard_debug_phase_times(shard, buf, n)
    if k < 0:
        _check(k)
    return list(buf)[:k]


def shard_debug_set_wait(shard: int, limit: int, skip_arrival: int = -1) -> None:
    """Test knob of the step kernel's bounded waits (include/shard_debug.h)."""
    _check(load_library().shard_debug_set_wait(shard, int(limit), int(skip_arrival)))


def shard_gemv_noalloc(shard: int, layer: int, op: int, x: int, M: int, y: int, y_ld: int, stream: int = 0,
                       check: bool = True) -> int:
    """One projection with the library's fixed scratch array (no device allocation)."""
    rc = load_library().shard_gemv_noalloc(shard, layer, op, x, M, y, y_ld, stream or None)
    return _check(rc) if check else rc


# ---------------------------------------------------------------------------
# LM head with the top-1 epilogue (include/head.h)
# ---------------------------------------------------------------------------

def head_create(hidden: int, vocab: int, group: int, rms_eps: float, lm_head, norm: np.ndarray) -> int:
    """lm_head: packed [vocab][hidden] matrix (.codes/.scales/.zeros arrays);
    norm: fp16 bits [hidden]."""
    cfg = head_config(hidden, vocab, group, 0, float(rms_eps))
    w = head_weights_host(shard_matrix_host(_np(lm_head.codes, np.uint8), _np(lm_head.scales, np.uint16),
                                            _np(lm_head.zeros, np.uint8)), _np(norm, np.uint16))
    out = ctypes.c_void_p()
    _check(load_library().head_create(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(out)))
    return out.value


def head_destroy(head: int) -> None:
    _check(load_library().head_destroy(head))


def head_top1(head: int, hidden: int, M: int, token: int, p_max: Optional[int], stream: int = 0,
              check: bool = True) -> int:
    """Device pointers as ints: hidden fp16 [M][H], token int32 [M], p_max fp32 [M] (or None)."""
    rc = load_library().head_top1(head, hidden, M, token, p_max or None, stream or None)
    return _check(rc) if check else rc


def head_top1_host(head: int, hidden: np.ndarray, stream: int = 0):
    """Host fp16 bits [M][H] -> (token int32 [M], p_max float32 [M])."""
    hidden = np.ascontiguousarray(hidden, dtype=np.uint16)
    M = hidden.shape[0]
    tok = np.empty(M, np.int32)
    p = np.empty(M, np.float32)
    _check(load_library().head_top1_host(head, _np(hidden), M, _np(tok), _np(p), stream or None))
    return tok, p


def head_debug_logits(head: int, hidden: int, M: int, logits: int, ld: int, stream: int = 0) -> None:
    _check(load_library().head_debug_logits(head, hidden, M, logits, ld, stream or None))
