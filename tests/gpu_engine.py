"""GPU engine for the shared scenario drivers: runs every call through the
C ABI of libshard (via the package's thin binding), with torch only holding
device buffers and providing the stream."""
from __future__ import annotations

import numpy as np
import torch

import paper_2608_19147_gb300 as pkg

TOL_REL_L2 = 1e-3   # relative L2 on fp16 hidden states
TOL_MAX_ABS = 2e-2  # max-abs on fp16 hidden states


def to_dev(a: np.ndarray, dtype=None) -> torch.Tensor:
    if a.dtype == np.uint16:
        a = a.view(np.int16)
    return torch.from_numpy(np.ascontiguousarray(a)).to("cuda")


class GpuShard:
    def __init__(self, shape, weights):
        self.shape = shape
        self.h = pkg.shard_create(pkg.make_config(shape), weights.layers, weights.embedding)

    def close(self):
        if self.h:
            pkg.shard_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class GpuEngine:
    def __init__(self, shard: GpuShard, n_rows: int, capacity: int):
        self.shard = shard
        self.shape = shard.shape
        self.st = pkg.kv_state_alloc(shard.h, n_rows, capacity)
        self.n_rows = n_rows

    @property
    def stream(self) -> int:
        return torch.cuda.current_stream().cuda_stream

    def step_raw(self, n_new, position_ids, mask, hidden_in=None, token_ids=None, beam_idx=None, check=True):
        M = int(sum(n_new))
        mask = np.ascontiguousarray(mask, dtype=np.uint8)
        if mask.ndim == 1:
            mask = mask.reshape(1, -1)
        d_mask = to_dev(mask)
        d_pos = to_dev(np.asarray(position_ids, dtype=np.int32))
        d_h = to_dev(hidden_in) if hidden_in is not None else None
        d_t = to_dev(np.asarray(token_ids, dtype=np.int32)) if token_ids is not None else None
        d_b = to_dev(np.asarray(beam_idx, dtype=np.int32)) if beam_idx is not None else None
        out = torch.empty((M, self.shape.hidden), dtype=torch.int16, device="cuda")
        rc = pkg.shard_step(self.shard.h, self.st, d_h.data_ptr() if d_h is not None else None,
                            d_t.data_ptr() if d_t is not None else None, list(n_new), d_pos.data_ptr(),
                            d_mask.data_ptr(), mask.shape[1], d_b.data_ptr() if d_b is not None else None,
                            out.data_ptr(), self.stream, check=check)
        keep = (d_mask, d_pos, d_h, d_t, d_b)  # alive until the sync below
        if rc != 0:
            return rc, None
        rc = pkg.shard_sync_status(self.shard.h, self.stream, check=check)
        del keep
        return rc, out.cpu().numpy().view(np.uint16)

    def step(self, n_new, position_ids, mask, hidden_in=None, token_ids=None, beam_idx=None):
        rc, out = self.step_raw(n_new, position_ids, mask, hidden_in, token_ids, beam_idx)
        return out

    def load(self, row, layer, k16, v16):
        pkg.kv_state_load(self.st, row, layer, k16, v16)

    def read(self, row, layer, start, n):
        return pkg.kv_state_read(self.st, row, layer, start, n, self.shape.n_kv_heads, self.shape.head_dim)

    def trim(self, row, keep):
        pkg.kv_trim(self.st, row, keep)

    def length(self, row):
        return pkg.kv_state_length(self.st, row)

    def close(self):
        if self.st:
            pkg.kv_state_free(self.st)
            self.st = None


def assert_close(got16: np.ndarray, want16: np.ndarray, rel=TOL_REL_L2, mx=TOL_MAX_ABS, what=""):
    g = got16.view(np.float16).astype(np.float64)
    w = want16.view(np.float16).astype(np.float64)
    assert np.isfinite(g).all(), what + ": non-finite GPU output"
    r = np.linalg.norm(g - w) / max(np.linalg.norm(w), 1e-30)
    m = np.abs(g - w).max()
    assert r <= rel and m <= mx, "%s: relL2 %.3e (tol %.1e) max-abs %.3e (tol %.1e)" % (what, r, rel, m, mx)
    return r, m
