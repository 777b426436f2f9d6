"""shard_gemv_noalloc: the projection entry point that allocates no device
memory, for callers that must not allocate while they run (a runtime that
has reserved all of HBM in its own pool, a thread that may not take the
allocator's lock, a loop that may not synchronise).  Its scratch is a fixed
device array inside the library; this checks, through the C ABI, that two
calls in a row give the same results as the allocating path
(shard_debug_gemv), and that oversized requests are refused.

Kept in its own file, collected last, so a failure here does not stop the
rest of a run with -x."""
import numpy as np
import pytest
import torch

import paper_2608_19147_gb300 as pkg
import synth

pytestmark = pytest.mark.gpu

SHAPES = [
    synth.TINY,
    synth.ShardShape("8b-1layer", 1, 4096, 32, 8, 128, 14336, 128, 0.02, 0, 1e-5, 500000.0, 4096),
]


def _run(fn, h, layer, op, x16, rows):
    M = x16.shape[0]
    dx = torch.from_numpy(np.ascontiguousarray(x16).view(np.int16)).cuda()
    y = torch.full((M, rows), float("nan"), dtype=torch.float32, device="cuda")
    fn(h, layer, op, dx.data_ptr(), M, y.data_ptr(), rows, torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    return y.cpu().numpy()


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: s.name)
def test_noalloc_matches_allocating_path_on_consecutive_calls(shape):
    w = synth.make_weights(shape, 11)
    h = pkg.shard_create(pkg.make_config(shape), w.layers, w.embedding)
    try:
        rng = np.random.default_rng(3)
        for M in (1, 5, 16):
            for op in range(4):
                rows, K, _ = pkg.shard_debug_op_info(h, 0, op)
                for call in range(2):  # two calls in a row reuse the same scratch
                    x16 = rng.standard_normal((M, K)).astype(np.float16).view(np.uint16)
                    want = _run(pkg.shard_debug_gemv, h, 0, op, x16, rows)
                    got = _run(pkg.shard_gemv_noalloc, h, 0, op, x16, rows)
                    assert np.isfinite(got).all()
                    scale = np.abs(want).max() + 1e-6
                    assert np.abs(got - want).max() <= 1e-5 * scale, (M, op, call)
    finally:
        pkg.shard_destroy(h)


def test_noalloc_refuses_requests_beyond_its_fixed_scratch():
    # a 160K-wide down projection: 16 padded activation rows alone need 5 MiB
    shape = synth.ShardShape("wide-ffn", 1, 64, 1, 1, 64, 163840, 128, 0.02, 0, 1e-5, 10000.0, 64)
    w = synth.make_weights(shape, 5)
    h = pkg.shard_create(pkg.make_config(shape), w.layers, w.embedding)
    try:
        rows, K, _ = pkg.shard_debug_op_info(h, 0, pkg.OP_DOWN)
        x = torch.zeros((16, K), dtype=torch.int16, device="cuda")
        y = torch.zeros((16, rows), dtype=torch.float32, device="cuda")
        rc = pkg.shard_gemv_noalloc(h, 0, pkg.OP_DOWN, x.data_ptr(), 16, y.data_ptr(), rows, check=False)
        assert rc == pkg.SHARD_ECAPACITY
        assert "scratch" in pkg.shard_last_error()
        # a single token fits
        x16 = np.random.default_rng(1).standard_normal((1, K)).astype(np.float16).view(np.uint16)
        want = _run(pkg.shard_debug_gemv, h, 0, pkg.OP_DOWN, x16, rows)
        got = _run(pkg.shard_gemv_noalloc, h, 0, pkg.OP_DOWN, x16, rows)
        assert np.abs(got - want).max() <= 1e-5 * (np.abs(want).max() + 1e-6)
    finally:
        pkg.shard_destroy(h)
