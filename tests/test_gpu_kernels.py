"""GPU parity of the projection kernel and the private weight layout, through
the C ABI: the layout read back is bit-exact with the oracle's dequantisation;
the GEMV is bit-exact on integer-valued inputs (every partial sum exact in
fp32) and within rounding of the oracle on random inputs, for M = 1..16."""
import numpy as np
import pytest
import torch

import oracle
import paper_2608_19147_gb300 as pkg
import synth

pytestmark = pytest.mark.gpu

SHAPES = {
    "tiny": synth.TINY,
    # one layer of the 8B stage: every projection shape of the workload
    "8b-1layer": synth.ShardShape("8b-1layer", 1, 4096, 32, 8, 128, 14336, 128, 0.02, 0, 1e-5, 500000.0, 4096),
    # ragged: K not a multiple of 128, F not a multiple of 8, group 64
    "ragged": synth.ShardShape("ragged", 1, 200, 4, 4, 64, 333, 64, 0.02, 0, 1e-5, 10000.0, 256),
}


def _natural_matrices(w, layer):
    """Source matrices of each fused projection, rows concatenated."""
    m = w.layers[layer].matrices
    return {pkg.OP_QKV: [m[0], m[1], m[2]], pkg.OP_O: [m[3]], pkg.OP_GU: [m[4], m[5]], pkg.OP_DOWN: [m[6]]}


@pytest.fixture(scope="module", params=list(SHAPES))
def shard(request):
    shape = SHAPES[request.param]
    w = synth.make_weights(shape, 99)
    h = pkg.shard_create(pkg.make_config(shape), w.layers, w.embedding)
    yield shape, w, h
    pkg.shard_destroy(h)


def test_unpack_is_bit_exact(shard):
    shape, w, h = shard
    for layer in range(shape.n_layers):
        mats = _natural_matrices(w, layer)
        for op in range(4):
            rows, K, _ = pkg.shard_debug_op_info(h, layer, op)
            out = torch.full((rows, K), float("nan"), dtype=torch.float32, device="cuda")
            pkg.shard_debug_unpack(h, layer, op, out.data_ptr(), K)
            want = np.concatenate([oracle.dequant(m) for m in mats[op]])
            got = out.cpu().numpy().astype(np.float64)
            assert np.array_equal(got, want), (layer, op)


def _gemv(h, layer, op, x16, rows):
    M = x16.shape[0]
    dx = torch.from_numpy(x16.view(np.int16)).cuda()
    y = torch.full((M, rows), float("nan"), dtype=torch.float32, device="cuda")
    pkg.shard_debug_gemv(h, layer, op, dx.data_ptr(), M, y.data_ptr(), rows, torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    return y.cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("M", [1, 2, 5, 8, 9, 16])
def test_gemv_random_matches_oracle(shard, M):
    shape, w, h = shard
    rng = np.random.default_rng(M)
    mats = _natural_matrices(w, 0)
    for op in range(4):
        rows, K, _ = pkg.shard_debug_op_info(h, 0, op)
        x16 = rng.standard_normal((M, K)).astype(np.float16)
        got = _gemv(h, 0, op, x16.view(np.uint16), rows)
        want = np.concatenate([oracle.gemv(m, x16.astype(np.float64)) for m in mats[op]], axis=1)
        # fp32 accumulation of exact products: error ~ 1e-7 relative to the row's magnitude
        scale = np.abs(x16.astype(np.float64)) @ np.abs(np.concatenate([oracle.dequant(m) for m in mats[op]])).T
        assert np.all(np.abs(got - want) <= 1e-5 * scale + 1e-6), (op, np.max(np.abs(got - want) / (scale + 1e-9)))


def _integer_weights(shape, seed):
    """Weights with power-of-two scales (2^-3 or 2^-4) so that products and
    sums of small-integer activations are exact in fp32."""
    rng = np.random.default_rng(seed)
    w = synth.make_weights(shape, seed)
    for lw in w.layers:
        for m in lw.matrices:
            m.scales[:] = rng.choice(np.array([2.0 ** -3, 2.0 ** -4], dtype=np.float16).view(np.uint16), m.scales.shape)
    return w


@pytest.mark.parametrize("M", [1, 3, 8, 16])
def test_gemv_integer_inputs_bit_exact(M):
    shape = SHAPES["8b-1layer"]
    w = _integer_weights(shape, 5)
    h = pkg.shard_create(pkg.make_config(shape), w.layers, w.embedding)
    try:
        rng = np.random.default_rng(M)
        mats = _natural_matrices(w, 0)
        for op in range(4):
            rows, K, _ = pkg.shard_debug_op_info(h, 0, op)
            x16 = rng.integers(-4, 5, (M, K)).astype(np.float16)
            got = _gemv(h, 0, op, x16.view(np.uint16), rows)
            want = np.concatenate([oracle.gemv(m, x16.astype(np.float64)) for m in mats[op]], axis=1)
            assert np.array_equal(got, want), op
    finally:
        pkg.shard_destroy(h)


def test_gemv_rows_independent_of_token_count(shard):
    # column m of an M-token product equals the single-token product bit for bit
    shape, w, h = shard
    rng = np.random.default_rng(1)
    rows, K, _ = pkg.shard_debug_op_info(h, 0, pkg.OP_GU)
    x16 = rng.standard_normal((16, K)).astype(np.float16).view(np.uint16)
    full = _gemv(h, 0, pkg.OP_GU, x16, rows)
    for m in (0, 7, 8, 15):
        one = _gemv(h, 0, pkg.OP_GU, np.ascontiguousarray(x16[m:m + 1]), rows)
        assert np.array_equal(one[0], full[m])
