"""Seeded synthetic inputs for the shard-decode workloads.

This package produces inputs only: Gaussian weights quantised to the packed
uint4 format that the shard boundary accepts, fp16 KV-cache prefills and
hidden states, token ids, speculative accept patterns and beam permutations.
It holds none of the shard forward's arithmetic.  Both the CUDA library's
tests/benchmark and the CPU oracle's tests draw their inputs from here, so
the two sides see identical bytes; neither side's code lives here.

The stand-in workloads follow the paper's Llama 3.1 shapes (Section 3.2
export, Section 6 evaluation, Section 6.11 70B deployment): the trained
weights and evaluation prompts are not available, so seeded Gaussian weights
and inputs of the same shapes stand in for them.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from dataclasses import dataclass, field
from typing import List, Optional, Tuple

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "synth.c")
_LIB = os.path.join(_HERE, "libsynth.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile libsynth.so with gcc if it is missing or older than synth.c."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-fPIC", "-shared", "-pthread", "-ffp-contract=off",
                               "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            u8p = ctypes.POINTER(ctypes.c_uint8)
            u16p = ctypes.POINTER(ctypes.c_uint16)
            u32p = ctypes.POINTER(ctypes.c_uint32)
            i32p = ctypes.POINTER(ctypes.c_int32)
            f32p = ctypes.POINTER(ctypes.c_float)
            f64p = ctypes.POINTER(ctypes.c_double)
            i64, u64, u32, c_int, c_double = (ctypes.c_int64, ctypes.c_uint64, ctypes.c_uint32,
                                              ctypes.c_int, ctypes.c_double)
            lib.synth_philox4x32_10.argtypes = [u32p, u32p, u32p]
            lib.synth_f64_to_f16.argtypes = [c_double]
            lib.synth_f64_to_f16.restype = ctypes.c_uint16
            lib.synth_f16_to_f64.argtypes = [ctypes.c_uint16]
            lib.synth_f16_to_f64.restype = c_double
            for name, p in (("synth_normal_f32", f32p), ("synth_normal_f16", u16p), ("synth_normal_f64", f64p)):
                getattr(lib, name).argtypes = [p, i64, c_double, c_double, u64, u32, u32, c_int]
            lib.synth_uniform_f64.argtypes = [f64p, i64, u64, u32, u32]
            lib.synth_uniform_int.argtypes = [i32p, i64, ctypes.c_int32, ctypes.c_int32, u64, u32, u32]
            lib.synth_quantize.argtypes = [f32p, c_int, c_int, c_int, u8p, u16p, u8p]
            lib.synth_quant_matrix.argtypes = [u8p, u16p, u8p, c_int, c_int, c_int, c_double, u64, u32, u32, c_int]
            _lib = lib
    return _lib


def _ptr(a: np.ndarray, ctype):
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.POINTER(ctype))


def default_threads() -> int:
    return max(1, min(64, os.cpu_count() or 1))


# ---------------------------------------------------------------------------
# Low-level generators
# ---------------------------------------------------------------------------

def philox4x32_10(ctr, key) -> np.ndarray:
    lib = _load()
    c = np.ascontiguousarray(ctr, dtype=np.uint32)
    k = np.ascontiguousarray(key, dtype=np.uint32)
    out = np.zeros(4, dtype=np.uint32)
    lib.synth_philox4x32_10(_ptr(c, ctypes.c_uint32), _ptr(k, ctypes.c_uint32), _ptr(out, ctypes.c_uint32))
    return out


def f64_to_f16_bits(x: float) -> int:
    return int(_load().synth_f64_to_f16(float(x)))


def normal(n: int, *, seed: int, stream: int, tag: int, mean: float = 0.0, sigma: float = 1.0,
           dtype=np.float32, threads: Optional[int] = None) -> np.ndarray:
    """n samples of N(mean, sigma^2); dtype float32, float64, or uint16 (fp16 bits)."""
    lib = _load()
    th = threads or default_threads()
    if dtype == np.float32:
        out = np.empty(n, dtype=np.float32)
        lib.synth_normal_f32(_ptr(out, ctypes.c_float), n, mean, sigma, seed, stream, tag, th)
    elif dtype == np.float64:
        out = np.empty(n, dtype=np.float64)
        lib.synth_normal_f64(_ptr(out, ctypes.c_double), n, mean, sigma, seed, stream, tag, th)
    elif dtype == np.uint16:
        out = np.empty(n, dtype=np.uint16)
        lib.synth_normal_f16(_ptr(out, ctypes.c_uint16), n, mean, sigma, seed, stream, tag, th)
    else:
        raise ValueError(dtype)
    return out


def uniform(n: int, *, seed: int, stream: int, tag: int) -> np.ndarray:
    out = np.empty(n, dtype=np.float64)
    _load().synth_uniform_f64(_ptr(out, ctypes.c_double), n, seed, stream, tag)
    return out


def uniform_int(n: int, lo: int, hi: int, *, seed: int, stream: int, tag: int) -> np.ndarray:
    """n integers uniform on [lo, hi] inclusive."""
    out = np.empty(n, dtype=np.int32)
    _load().synth_uniform_int(_ptr(out, ctypes.c_int32), n, lo, hi, seed, stream, tag)
    return out


@dataclass
class PackedMatrix:
    """One uint4 group-quantised matrix in the boundary's packed format."""
    rows: int
    cols: int
    group: int
    codes: np.ndarray   # uint8 [rows][ceil(cols/2)], low nibble = even column
    scales: np.ndarray  # uint16 (fp16 bits) [rows][G]
    zeros: np.ndarray   # uint8 [rows][ceil(G/2)], low nibble = even group

    @property
    def n_groups(self) -> int:
        return (self.cols + self.group - 1) // self.group

    def nbytes(self) -> int:
        return self.codes.nbytes + self.scales.nbytes + self.zeros.nbytes


def _empty_packed(rows: int, cols: int, group: int) -> PackedMatrix:
    G = (cols + group - 1) // group
    return PackedMatrix(rows, cols, group,
                        np.zeros((rows, (cols + 1) // 2), dtype=np.uint8),
                        np.zeros((rows, G), dtype=np.uint16),
                        np.zeros((rows, (G + 1) // 2), dtype=np.uint8))


def quantize(w: np.ndarray, group: int) -> PackedMatrix:
    """Asymmetric uint4 min-max quantisation of a given fp32 matrix."""
    w = np.ascontiguousarray(w, dtype=np.float32)
    rows, cols = w.shape
    m = _empty_packed(rows, cols, group)
    _load().synth_quantize(_ptr(w, ctypes.c_float), rows, cols, group, _ptr(m.codes, ctypes.c_uint8),
                           _ptr(m.scales, ctypes.c_uint16), _ptr(m.zeros, ctypes.c_uint8))
    return m


def quant_matrix(rows: int, cols: int, group: int, sigma: float, *, seed: int, stream: int, tag: int,
                 threads: Optional[int] = None) -> PackedMatrix:
    """Weights N(0, sigma^2) drawn in fp32, quantised and packed."""
    m = _empty_packed(rows, cols, group)
    _load().synth_quant_matrix(_ptr(m.codes, ctypes.c_uint8), _ptr(m.scales, ctypes.c_uint16),
                               _ptr(m.zeros, ctypes.c_uint8), rows, cols, group, sigma, seed, stream, tag,
                               threads or default_threads())
    return m


# ---------------------------------------------------------------------------
# Shard shapes (Llama-style layer ranges) and their seeded weights
# ---------------------------------------------------------------------------

MATRIX_NAMES = ("q", "k", "v", "o", "gate", "up", "down")

TAG_WEIGHT, TAG_NORM, TAG_EMBED, TAG_KV, TAG_HIDDEN, TAG_TOKENS, TAG_ACCEPT, TAG_BEAM, TAG_LENGTHS, TAG_DRAFT = range(1, 11)
TAG_HEAD = 11


@dataclass(frozen=True)
class ShardShape:
    name: str
    n_layers: int
    hidden: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    group: int
    weight_sigma: float
    vocab: int = 0            # > 0: the shard owns the token embedding (first stage)
    rms_eps: float = 1e-5
    rope_theta: float = 500000.0
    max_position: int = 8192  # size of the precomputed rotary table

    def matrix_shape(self, name: str) -> Tuple[int, int]:
        H, dq, dkv, F = self.hidden, self.n_heads * self.head_dim, self.n_kv_heads * self.head_dim, self.ffn
        return {"q": (dq, H), "k": (dkv, H), "v": (dkv, H), "o": (H, dq),
                "gate": (F, H), "up": (F, H), "down": (H, F)}[name]

    def params_per_layer(self) -> int:
        return sum(r * c for r, c in (self.matrix_shape(n) for n in MATRIX_NAMES))

    def packed_bytes_per_layer(self) -> int:
        """Bytes of codes + fp16 scales + uint4 zeros per layer (algorithmic, unpadded)."""
        total = 0
        for n in MATRIX_NAMES:
            r, c = self.matrix_shape(n)
            G = -(-c // self.group)
            total += r * c / 2 + r * G * 2 + r * G / 2
        return int(total)

    def kv_bytes_per_token(self) -> int:
        """fp16 K and V bytes per cached token per layer."""
        return 2 * 2 * self.n_kv_heads * self.head_dim


TINY = ShardShape("tiny-2L-h256", n_layers=2, hidden=256, n_heads=4, n_kv_heads=2, head_dim=64, ffn=688,
                  group=32, weight_sigma=0.02, vocab=512, max_position=1024)
LLAMA8B_STAGE = ShardShape("llama3.1-8b-stage1of2-16L", n_layers=16, hidden=4096, n_heads=32, n_kv_heads=8,
                           head_dim=128, ffn=14336, group=128, weight_sigma=0.02, vocab=128256, max_position=4096)
LLAMA70B_STAGE = ShardShape("llama3.1-70b-stage1of4-20L", n_layers=20, hidden=8192, n_heads=64, n_kv_heads=8,
                            head_dim=128, ffn=28672, group=128, weight_sigma=0.015, vocab=0, max_position=8192)


@dataclass
class LayerWeights:
    matrices: List[PackedMatrix]   # q, k, v, o, gate, up, down
    attn_norm: np.ndarray          # uint16 fp16 bits [H]
    ffn_norm: np.ndarray           # uint16 fp16 bits [H]


@dataclass
class ShardWeights:
    shape: ShardShape
    seed: int
    layers: List[LayerWeights] = field(default_factory=list)
    embedding: Optional[np.ndarray] = None  # uint16 fp16 bits [V][H]

    def packed_bytes(self) -> int:
        return sum(m.nbytes() for lw in self.layers for m in lw.matrices)


def layer_weights(shape: ShardShape, seed: int, layer: int, threads: Optional[int] = None) -> LayerWeights:
    """The seeded weights of one layer of a shard (its own streams: the same
    values whether the layer is made alone or as part of the whole shard)."""
    mats = []
    for mi, name in enumerate(MATRIX_NAMES):
        r, c = shape.matrix_shape(name)
        mats.append(quant_matrix(r, c, shape.group, shape.weight_sigma, seed=seed,
                                 stream=layer * 16 + mi, tag=TAG_WEIGHT, threads=threads))
    an = normal(shape.hidden, seed=seed, stream=layer * 2, tag=TAG_NORM, mean=1.0, sigma=0.1, dtype=np.uint16)
    fn = normal(shape.hidden, seed=seed, stream=layer * 2 + 1, tag=TAG_NORM, mean=1.0, sigma=0.1, dtype=np.uint16)
    return LayerWeights(mats, an, fn)


def embedding(shape: ShardShape, seed: int, threads: Optional[int] = None) -> np.ndarray:
    """The seeded token embedding of a first-stage shard (fp16 N(0,1) bits [V][H])."""
    return normal(shape.vocab * shape.hidden, seed=seed, stream=0, tag=TAG_EMBED,
                  dtype=np.uint16, threads=threads).reshape(shape.vocab, shape.hidden)


def make_weights(shape: ShardShape, seed: int, threads: Optional[int] = None, n_layers: Optional[int] = None) -> ShardWeights:
    """Seeded weights for a shard: per layer q,k,v,o,gate,up,down ~ N(0, sigma^2)
    quantised to uint4 (group = shape.group); norm weights fp16(1 + 0.1 N(0,1));
    embedding (when vocab > 0) fp16 N(0,1)."""
    sw = ShardWeights(shape, seed)
    L = shape.n_layers if n_layers is None else n_layers
    for layer in range(L):
        sw.layers.append(layer_weights(shape, seed, layer, threads))
    if shape.vocab > 0:
        sw.embedding = embedding(shape, seed, threads)
    return sw


@dataclass
class HeadWeights:
    """The final stage's LM head: final RMSNorm weight and the [V][H] lm_head."""
    hidden: int
    vocab: int
    group: int
    lm_head: PackedMatrix          # [vocab][hidden]
    norm: np.ndarray               # uint16 fp16 bits [hidden]
    rms_eps: float = 1e-5

    def packed_bytes(self) -> int:
        return self.lm_head.nbytes()


def make_head(hidden: int, vocab: int, group: int, seed: int, sigma: float = 0.02, rms_eps: float = 1e-5,
              threads: Optional[int] = None) -> HeadWeights:
    """Seeded LM head: lm_head ~ N(0, sigma^2) quantised to uint4 like the
    layer matrices; final norm weight fp16(1 + 0.1 N(0,1))."""
    w = quant_matrix(vocab, hidden, group, sigma, seed=seed, stream=0, tag=TAG_HEAD, threads=threads)
    norm = normal(hidden, seed=seed, stream=1, tag=TAG_HEAD, mean=1.0, sigma=0.1, dtype=np.uint16)
    return HeadWeights(hidden, vocab, group, w, norm, rms_eps)


# ---------------------------------------------------------------------------
# Per-step inputs
# ---------------------------------------------------------------------------

def kv_prefill(shape: ShardShape, seed: int, row: int, length: int, layer: int) -> Tuple[np.ndarray, np.ndarray]:
    """fp16 N(0,1) K and V for one cache row and layer, layout [length][Hkv][d] (uint16 bits)."""
    n = length * shape.n_kv_heads * shape.head_dim
    k = normal(n, seed=seed, stream=(row << 16) | (layer << 1), tag=TAG_KV, dtype=np.uint16)
    v = normal(n, seed=seed, stream=(row << 16) | (layer << 1) | 1, tag=TAG_KV, dtype=np.uint16)
    return (k.reshape(length, shape.n_kv_heads, shape.head_dim), v.reshape(length, shape.n_kv_heads, shape.head_dim))


def hidden_in(shape: ShardShape, seed: int, step: int, M: int) -> np.ndarray:
    """fp16 N(0,1) hidden states [M][H] (uint16 bits)."""
    return normal(M * shape.hidden, seed=seed, stream=step, tag=TAG_HIDDEN, dtype=np.uint16).reshape(M, shape.hidden)


def token_ids(shape: ShardShape, seed: int, step: int, M: int) -> np.ndarray:
    """Token ids uniform on [0, vocab)."""
    return uniform_int(M, 0, shape.vocab - 1, seed=seed, stream=step, tag=TAG_TOKENS)


def accepted_drafts(seed: int, step: int, k: int = 4, p: float = 0.6) -> int:
    """Greedy longest-prefix acceptance stand-in: k Bernoulli(p) draws, the
    number of leading successes is the number of accepted drafts."""
    u = uniform(k, seed=seed, stream=step, tag=TAG_ACCEPT)
    a = 0
    while a < k and u[a] < p:
        a += 1
    return a


def permutation(seed: int, step: int, n: int) -> np.ndarray:
    """Uniform random permutation of range(n) (Fisher-Yates on seeded uniforms)."""
    perm = np.arange(n, dtype=np.int32)
    for i in range(n - 1, 0, -1):
        j = int(uniform_int(1, 0, i, seed=seed, stream=step * 64 + i, tag=TAG_BEAM)[0])
        perm[i], perm[j] = perm[j], perm[i]
    return perm


def lengths(seed: int, n: int, lo: int, hi: int) -> np.ndarray:
    """n cache lengths uniform on [lo, hi]."""
    return uniform_int(n, lo, hi, seed=seed, stream=0, tag=TAG_LENGTHS)


def draft_tokens(seed: int, step: int, n: int, vocab: int) -> np.ndarray:
    """Seeded token ids used as deliberately wrong draft proposals."""
    return uniform_int(n, 0, vocab - 1, seed=seed, stream=step, tag=TAG_DRAFT)
