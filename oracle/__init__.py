"""ORACLE -- test infrastructure, not part of the product.

ctypes binding of oracle.c: a plain fp64 CPU implementation of the decode
step of one pipeline shard (stateful KV cache with the beam_idx gather of
Section 4 and the attention-mask rewind of Section 5.2 of the paper).  Only
tests, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline leg use
it.  It shares no code with the CUDA library and imports nothing from it.

Objects are duck-typed: a ``shape`` needs n_layers, hidden, n_heads,
n_kv_heads, head_dim, ffn, group, vocab, rms_eps, rope_theta; ``weights``
needs ``layers`` (each with ``matrices`` of codes/scales/zeros arrays and
``attn_norm``/``ffn_norm``) and ``embedding``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from typing import Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

OK, EINVAL, ECAP, ENOMEM = 0, -1, -2, -3


def build(force: bool = False) -> str:
    """Compile liboracle.so with gcc (OpenMP over output rows) if stale."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off",
                               "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


class _Config(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("hidden", ctypes.c_int32), ("n_heads", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32), ("ffn", ctypes.c_int32),
                ("group", ctypes.c_int32), ("vocab", ctypes.c_int32),
                ("rms_eps", ctypes.c_double), ("rope_theta", ctypes.c_double)]


class _Matrix(ctypes.Structure):
    _fields_ = [("codes", ctypes.c_void_p), ("scales", ctypes.c_void_p), ("zeros", ctypes.c_void_p)]


class _Layer(ctypes.Structure):
    _fields_ = [("w", _Matrix * 7), ("attn_norm", ctypes.c_void_p), ("ffn_norm", ctypes.c_void_p)]


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            vp, ip, dp = ctypes.c_void_p, ctypes.c_int, ctypes.c_double
            lib.or_f16_to_f64.argtypes = [ctypes.c_uint16]
            lib.or_f16_to_f64.restype = dp
            lib.or_f64_to_f16.argtypes = [dp]
            lib.or_f64_to_f16.restype = ctypes.c_uint16
            lib.or_round_f16.argtypes = [dp]
            lib.or_round_f16.restype = dp
            lib.or_set_threads.argtypes = [ip]
            lib.or_get_threads.restype = ip
            lib.or_dequant.argtypes = [ctypes.POINTER(_Matrix), ip, ip, ip, vp]
            lib.or_gemv.argtypes = [ctypes.POINTER(_Matrix), ip, ip, ip, vp, ip, vp]
            lib.or_rmsnorm.argtypes = [vp, ip, vp, dp, vp]
            lib.or_rope.argtypes = [vp, ip, ip, dp]
            lib.or_silu.argtypes = [dp]
            lib.or_silu.restype = dp
            lib.or_attend.argtypes = [vp, vp, vp, ip, ip, ip, vp, vp]
            lib.or_attend.restype = ip
            lib.or_shard_create.argtypes = [ctypes.POINTER(_Config), ctypes.POINTER(_Layer), vp]
            lib.or_shard_create.restype = vp
            lib.or_shard_destroy.argtypes = [vp]
            lib.or_state_create.argtypes = [vp, ip, ip]
            lib.or_state_create.restype = vp
            lib.or_state_destroy.argtypes = [vp]
            lib.or_state_length.argtypes = [vp, ip]
            lib.or_state_length.restype = ip
            lib.or_state_load.argtypes = [vp, ip, ip, vp, vp, ip]
            lib.or_state_load.restype = ip
            lib.or_state_read.argtypes = [vp, ip, ip, ip, ip, vp, vp, vp, vp]
            lib.or_state_read.restype = ip
            lib.or_trim.argtypes = [vp, ip, vp, ip]
            lib.or_trim.restype = ip
            lib.or_step.argtypes = [vp, vp, vp, vp, vp, ip, vp, vp, ip, vp, ip, vp, vp]
            lib.or_step.restype = ip
            lib.or_step_packed.argtypes = [vp, vp, vp, vp, ip, vp, vp, ip, ip, vp, vp]
            lib.or_step_packed.restype = ip
            lib.or_logits.argtypes = [vp, ip, ip, vp, ip, dp, vp]
            lib.or_head_top1.argtypes = [vp, ip, ip, vp, dp, ctypes.POINTER(_Matrix), ip, ip, ip, vp, vp, vp, vp]
            _lib = lib
    return _lib


def _p(a: Optional[np.ndarray]):
    if a is None:
        return None
    assert a.flags["C_CONTIGUOUS"], "array must be C-contiguous"
    return a.ctypes.data


def set_threads(n: int) -> None:
    _load().or_set_threads(int(n))


def get_threads() -> int:
    return int(_load().or_get_threads())


# ---------------------------------------------------------------------------
# Building blocks (exposed for the oracle's own pin tests)
# ---------------------------------------------------------------------------

def f16_round(x: float) -> float:
    return float(_load().or_round_f16(float(x)))


def f64_to_f16_bits(x: float) -> int:
    return int(_load().or_f64_to_f16(float(x)))


def f16_bits_to_f64(h: int) -> float:
    return float(_load().or_f16_to_f64(int(h)))


def _matrix_struct(m) -> _Matrix:
    return _Matrix(_p(m.codes), _p(m.scales), _p(m.zeros))


def dequant(m) -> np.ndarray:
    """Dense fp64 [rows][cols] of a packed matrix: W = (q - z) * s."""
    out = np.empty((m.rows, m.cols), dtype=np.float64)
    ms = _matrix_struct(m)
    _load().or_dequant(ctypes.byref(ms), m.rows, m.cols, m.group, _p(out))
    return out


def gemv(m, x: np.ndarray) -> np.ndarray:
    """y[t] = W x[t] for x [M][cols] (fp64)."""
    x = np.ascontiguousarray(x, dtype=np.float64).reshape(-1, m.cols)
    y = np.empty((x.shape[0], m.rows), dtype=np.float64)
    ms = _matrix_struct(m)
    _load().or_gemv(ctypes.byref(ms), m.rows, m.cols, m.group, _p(x), x.shape[0], _p(y))
    return y


def rmsnorm(x: np.ndarray, w16: Optional[np.ndarray], eps: float) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float64)
    out = np.empty_like(x)
    w = None if w16 is None else np.ascontiguousarray(w16, dtype=np.uint16)
    _load().or_rmsnorm(_p(x), x.size, _p(w), eps, _p(out))
    return out


def rope(vec: np.ndarray, pos: int, theta: float) -> np.ndarray:
    v = np.array(vec, dtype=np.float64, copy=True)
    _load().or_rope(_p(v), v.size, int(pos), float(theta))
    return v


def silu(x: float) -> float:
    return float(_load().or_silu(float(x)))


def attend(q: np.ndarray, K: np.ndarray, V: np.ndarray, visible: np.ndarray) -> np.ndarray:
    """Softmax attention of one query over rows of K/V where visible != 0."""
    q = np.ascontiguousarray(q, dtype=np.float64)
    K = np.ascontiguousarray(K, dtype=np.float64)
    V = np.ascontiguousarray(V, dtype=np.float64)
    vis = np.ascontiguousarray(visible, dtype=np.uint8)
    out = np.empty(q.size, dtype=np.float64)
    _load().or_attend(_p(q), _p(K), _p(V), K.shape[0], K.shape[1], q.size, _p(vis), _p(out))
    return out


def logits(h: np.ndarray, embedding: np.ndarray, eps: float) -> np.ndarray:
    """Test head: tied-embedding logits after an un-weighted RMSNorm."""
    h = np.ascontiguousarray(h, dtype=np.float64)
    M, H = h.shape
    E = np.ascontiguousarray(embedding, dtype=np.uint16)
    out = np.empty((M, E.shape[0]), dtype=np.float64)
    _load().or_logits(_p(h), M, H, _p(E), E.shape[0], eps, _p(out))
    return out


def head_top1(h16: np.ndarray, norm16: np.ndarray, w, eps: float, round_points: bool = True):
    """LM head with the top-1 epilogue (Section 6.7): fp16 hidden rows
    [M][H] -> (token [M] int32, p_max [M], margin [M], logits [M][V]), all
    fp64 but the token; w is the [V][H] packed INT4 lm_head (.codes,
    .scales, .zeros, .rows, .cols, .group)."""
    h16 = np.ascontiguousarray(h16, dtype=np.uint16)
    M, H = h16.shape
    assert w.cols == H
    V = w.rows
    norm16 = np.ascontiguousarray(norm16, dtype=np.uint16)
    tok = np.empty(M, np.int32)
    p = np.empty(M, np.float64)
    margin = np.empty(M, np.float64)
    lg = np.empty((M, V), np.float64)
    m = _matrix_struct(w)
    _load().or_head_top1(_p(h16), M, H, _p(norm16), eps, ctypes.byref(m), V, w.group, int(round_points), _p(tok),
                         _p(p), _p(margin), _p(lg))
    return tok, p, margin, lg


# ---------------------------------------------------------------------------
# Shard and KV state
# ---------------------------------------------------------------------------

class OracleShard:
    def __init__(self, shape, weights):
        lib = _load()
        self.shape = shape
        self._weights = weights  # keep arrays alive
        cfg = _Config(shape.n_layers, shape.hidden, shape.n_heads, shape.n_kv_heads, shape.head_dim, shape.ffn,
                      shape.group, shape.vocab if weights.embedding is not None else 0,
                      float(shape.rms_eps), float(shape.rope_theta))
        L = len(weights.layers)
        if L != shape.n_layers:
            raise ValueError("weights have %d layers, shape %d" % (L, shape.n_layers))
        layers = (_Layer * L)()
        for i, lw in enumerate(weights.layers):
            for j, m in enumerate(lw.matrices):
                layers[i].w[j] = _matrix_struct(m)
            layers[i].attn_norm = _p(lw.attn_norm)
            layers[i].ffn_norm = _p(lw.ffn_norm)
        self._layers = layers
        self._cfg = cfg
        self._h = lib.or_shard_create(ctypes.byref(cfg), layers, _p(weights.embedding))
        if not self._h:
            raise ValueError("or_shard_create rejected the configuration")

    def __del__(self):
        if getattr(self, "_h", None):
            _load().or_shard_destroy(self._h)
            self._h = None

    def state(self, n_rows: int, capacity: int) -> "OracleState":
        return OracleState(self, n_rows, capacity)


class OracleState:
    def __init__(self, shard: OracleShard, n_rows: int, capacity: int):
        self.shard = shard
        self.n_rows, self.capacity = n_rows, capacity
        self._h = _load().or_state_create(shard._h, n_rows, capacity)
        if not self._h:
            raise MemoryError("or_state_create failed")

    def __del__(self):
        if getattr(self, "_h", None):
            _load().or_state_destroy(self._h)
            self._h = None

    def length(self, row: int) -> int:
        return int(_load().or_state_length(self._h, row))

    def load(self, row: int, layer: int, k16: np.ndarray, v16: np.ndarray) -> int:
        k = np.ascontiguousarray(k16, dtype=np.uint16)
        v = np.ascontiguousarray(v16, dtype=np.uint16)
        return int(_load().or_state_load(self._h, row, layer, _p(k), _p(v), k.shape[0]))

    def read(self, row: int, layer: int, start: int, n: int, f64: bool = False):
        s = self.shard.shape
        shp = (n, s.n_kv_heads, s.head_dim)
        if f64:
            k = np.empty(shp, dtype=np.float64)
            v = np.empty(shp, dtype=np.float64)
            rc = _load().or_state_read(self._h, row, layer, start, n, None, None, _p(k), _p(v))
        else:
            k = np.empty(shp, dtype=np.uint16)
            v = np.empty(shp, dtype=np.uint16)
            rc = _load().or_state_read(self._h, row, layer, start, n, _p(k), _p(v), None, None)
        if rc != OK:
            raise ValueError("or_state_read failed: %d" % rc)
        return k, v

    def trim(self, row: int, keep: np.ndarray) -> int:
        keep = np.ascontiguousarray(keep, dtype=np.uint8)
        return int(_load().or_trim(self._h, row, _p(keep), keep.size))

    def step(self, n_new: Sequence[int], position_ids: np.ndarray, mask: np.ndarray, *,
             hidden_in: Optional[np.ndarray] = None, token_ids: Optional[np.ndarray] = None,
             beam_idx: Optional[np.ndarray] = None, round_points: bool = True, want_f64: bool = False):
        """One decode step. Returns (rc, out16 [M][H] uint16, out64 or None)."""
        s = self.shard.shape
        n = np.ascontiguousarray(n_new, dtype=np.int32)
        M = int(n.sum())
        pos = np.ascontiguousarray(position_ids, dtype=np.int32)
        msk = np.ascontiguousarray(mask, dtype=np.uint8)
        if msk.ndim == 1:
            msk = msk.reshape(1, -1)
        hid = None if hidden_in is None else np.ascontiguousarray(hidden_in, dtype=np.uint16)
        tok = None if token_ids is None else np.ascontiguousarray(token_ids, dtype=np.int32)
        beam = None if beam_idx is None else np.ascontiguousarray(beam_idx, dtype=np.int32)
        out16 = np.zeros((M, s.hidden), dtype=np.uint16)
        out64 = np.zeros((M, s.hidden), dtype=np.float64) if want_f64 else None
        rc = _load().or_step(self.shard._h, self._h, _p(hid), _p(tok), _p(n), len(n), _p(pos), _p(msk),
                             msk.shape[1], _p(beam), 1 if round_points else 0, _p(out16), _p(out64))
        return int(rc), out16, out64

    def step_packed(self, position_ids: np.ndarray, mask2d: np.ndarray, *, hidden_in: Optional[np.ndarray] = None,
                    token_ids: Optional[np.ndarray] = None, round_points: bool = True, want_f64: bool = False):
        """Packed step (Section 8.6): S rows on cache row 0, token t seeing
        the entries j with mask2d[t][j] != 0.  Returns (rc, out16, out64)."""
        s = self.shard.shape
        pos = np.ascontiguousarray(position_ids, dtype=np.int32)
        S = int(pos.size)
        msk = np.ascontiguousarray(mask2d, dtype=np.uint8)
        assert msk.ndim == 2 and msk.shape[0] == S
        hid = None if hidden_in is None else np.ascontiguousarray(hidden_in, dtype=np.uint16)
        tok = None if token_ids is None else np.ascontiguousarray(token_ids, dtype=np.int32)
        out16 = np.zeros((S, s.hidden), dtype=np.uint16)
        out64 = np.zeros((S, s.hidden), dtype=np.float64) if want_f64 else None
        rc = _load().or_step_packed(self.shard._h, self._h, _p(hid), _p(tok), S, _p(pos), _p(msk), msk.shape[1],
                                    1 if round_points else 0, _p(out16), _p(out64))
        return int(rc), out16, out64
