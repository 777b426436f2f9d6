"""GPU parity of the many-token tensor-core projection (tcgen05,
shard_debug_gemm) against the fp64 oracle, through the C ABI: for token
counts that fill one, several and ragged token tiles, every projection of
the tiny shard (group 32), one 8B layer (group 128) and a ragged shape
(group 64, K not a multiple of 128, F not a multiple of 8) is within the
fp32 accumulation bound of the oracle; with integer activations and
power-of-two scales (every sum exact in fp32) it is bit-exact; and it
equals the decode step's GEMV where both are exact."""
import numpy as np
import pytest
import torch

import oracle
import paper_2608_19147_gb300 as pkg
import synth

pytestmark = pytest.mark.gpu

SHAPES = {
    "tiny": synth.TINY,
    "8b-1layer": synth.ShardShape("8b-1layer", 1, 4096, 32, 8, 128, 14336, 128, 0.02, 0, 1e-5, 500000.0, 4096),
    "ragged": synth.ShardShape("ragged", 1, 200, 4, 4, 64, 333, 64, 0.02, 0, 1e-5, 10000.0, 256),
}


def _mats(w):
    m = w.layers[0].matrices
    return {pkg.OP_QKV: [m[0], m[1], m[2]], pkg.OP_O: [m[3]], pkg.OP_GU: [m[4], m[5]], pkg.OP_DOWN: [m[6]]}


def _gemm(h, op, x16, rows):
    S, K = x16.shape
    ld = (K + 127) // 128 * 128
    xp = np.zeros((S, ld), np.uint16)
    xp[:, :K] = x16
    dx = torch.from_numpy(xp.view(np.int16)).cuda()
    y = torch.full((S, rows), float("nan"), dtype=torch.float32, device="cuda")
    pkg.shard_debug_gemm(h, 0, op, dx.data_ptr(), ld, S, y.data_ptr(), rows, torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    return y.cpu().numpy().astype(np.float64)


@pytest.fixture(scope="module", params=list(SHAPES))
def shard(request):
    shape = SHAPES[request.param]
    w = synth.make_weights(shape, 99)
    h = pkg.shard_create(pkg.make_config(shape), w.layers, w.embedding)
    yield shape, w, h
    pkg.shard_destroy(h)


@pytest.mark.parametrize("S", [1, 16, 33, 128, 300])
def test_gemm_matches_oracle(shard, S):
    shape, w, h = shard
    rng = np.random.default_rng(S)
    mats = _mats(w)
    for op in range(4):
        rows, K, _ = pkg.shard_debug_op_info(h, 0, op)
        x16 = rng.standard_normal((S, K)).astype(np.float16)
        got = _gemm(h, op, x16.view(np.uint16), rows)
        want = np.concatenate([oracle.gemv(m, x16.astype(np.float64)) for m in mats[op]], axis=1)
        scale = np.abs(x16.astype(np.float64)) @ np.abs(np.concatenate([oracle.dequant(m) for m in mats[op]])).T
        assert np.isfinite(got).all(), op
        assert np.all(np.abs(got - want) <= 1e-5 * scale + 1e-6), (op, np.max(np.abs(got - want) / (scale + 1e-9)))


def test_gemm_integer_inputs_bit_exact_and_equal_to_the_gemv():
    shape = SHAPES["8b-1layer"]
    rng = np.random.default_rng(5)
    w = synth.make_weights(shape, 5)
    for lw in w.layers:
        for m in lw.matrices:
            m.scales[:] = rng.choice(np.array([2.0 ** -3, 2.0 ** -4], dtype=np.float16).view(np.uint16), m.scales.shape)
    h = pkg.shard_create(pkg.make_config(shape), w.layers, w.embedding)
    try:
        mats = _mats(w)
        for op in range(4):
            rows, K, _ = pkg.shard_debug_op_info(h, 0, op)
            x16 = rng.integers(-4, 5, (40, K)).astype(np.float16)
            got = _gemm(h, op, x16.view(np.uint16), rows)
            want = np.concatenate([oracle.gemv(m, x16.astype(np.float64)) for m in mats[op]], axis=1)
            assert np.array_equal(got, want), op
            dx = torch.from_numpy(x16[:16].view(np.int16)).cuda()
            y = torch.empty((16, rows), dtype=torch.float32, device="cuda")
            pkg.shard_debug_gemv(h, 0, op, dx.data_ptr(), 16, y.data_ptr(), rows,
                                 torch.cuda.current_stream().cuda_stream)
            torch.cuda.synchronize()
            assert np.array_equal(y.cpu().numpy().astype(np.float64), got[:16]), op
    finally:
        pkg.shard_destroy(h)
