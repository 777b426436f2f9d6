"""shard_gemv_noalloc: the projection entry point that allocates no device
memory, for callers that must not allocate while they run (a runtime that
has reserved all of HBM in its own pool, a thread that may not take the
allocator's lock, a loop that may not synchronise).  Its scratch is a fixed
device array inside the library.  Through the C ABI, on two calls in a row:
the results match the fp64 oracle's projection within the fp32 rounding the
other GEMV tests allow, and equal the allocating path (shard_debug_gemv) bit
for bit (both add their partial sums in 64-bit fixed point, so the order of
arrival does not matter); the call leaves no error behind in the shard's
status word; and oversized requests are refused.

Kept in its own file, collected last, so a failure here does not stop the
rest of a run with -x."""
import numpy as np
import pytest
import torch

import oracle
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
        m = w.layers[0].matrices
        mats = {pkg.OP_QKV: [m[0], m[1], m[2]], pkg.OP_O: [m[3]], pkg.OP_GU: [m[4], m[5]], pkg.OP_DOWN: [m[6]]}
        for M in (1, 5, 16):
            for op in range(4):
                rows, K, _ = pkg.shard_debug_op_info(h, 0, op)
                dense = np.concatenate([oracle.dequant(mm) for mm in mats[op]])
                for call in range(2):  # two calls in a row reuse the same scratch
                    x16 = rng.standard_normal((M, K)).astype(np.float16)
                    got = _run(pkg.shard_gemv_noalloc, h, 0, op, x16.view(np.uint16), rows)
                    want = _run(pkg.shard_debug_gemv, h, 0, op, x16.view(np.uint16), rows)
                    assert np.array_equal(got, want), (M, op, call)
                    ref = np.concatenate([oracle.gemv(mm, x16.astype(np.float64)) for mm in mats[op]], axis=1)
                    # fp32 accumulation of exact products, as in the other GEMV tests
                    scale = np.abs(x16.astype(np.float64)) @ np.abs(dense).T
                    assert np.all(np.abs(got - ref) <= 1e-5 * scale + 1e-6), (M, op, call)
        assert pkg.shard_sync_status(h, torch.cuda.current_stream().cuda_stream, check=False) == pkg.SHARD_OK
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
        assert np.array_equal(got, want)
    finally:
        pkg.shard_destroy(h)
