"""The step kernel's cross-CTA waits are bounded: a wait that runs out sets a
status bit and the kernel finishes instead of hanging the GPU.  This test
makes one run out on purpose -- without faulting or hanging anything: a test
knob (shard_debug_set_wait) shortens the poll limit and makes CTA 1 leave out
one grid-barrier arrival, so every other CTA's wait at that barrier gives
up -- and checks, through the C ABI, that

* the step returns promptly and is reported as "pipeline wait timed out"
  (EINVAL) by shard_sync_status;
* the KV state stays rejected (the next step is refused) until it is reset;
* after a reset, with the knob off, the next step is correct again (it
  matches the oracle) -- the library put its work buffers back in order.
"""
import time

import numpy as np
import pytest

import paper_2608_19147_gb300 as pkg
import synth
from gpu_engine import GpuEngine, GpuShard, assert_close
from scenarios import OracleEngine, prefill

pytestmark = pytest.mark.gpu
TINY = synth.TINY
SEED = 424242


def test_a_wait_that_runs_out_is_reported_and_the_state_recovers():
    w = synth.make_weights(TINY, SEED)
    sh = GpuShard(TINY, w)
    g = GpuEngine(sh, 1, 96)
    try:
        prefill(g, TINY, SEED, 0, 40)
        h = synth.hidden_in(TINY, SEED, 0, 1)
        args = ([1], np.array([40], np.int32), np.ones(41, np.uint8))
        # CTA 1 skips arrival 2 (the end of layer 0's o projection)
        pkg.shard_debug_set_wait(sh.h, 1 << 12, 2)
        t0 = time.time()
        rc, _ = g.step_raw(*args, hidden_in=h, check=False)
        elapsed = time.time() - t0
        assert rc == pkg.SHARD_EINVAL, rc
        assert "timed out" in pkg.shard_last_error()
        assert elapsed < 10.0, elapsed
        # the state stays rejected until it is reset
        pkg.shard_debug_set_wait(sh.h, 1 << 22, -1)
        rc, _ = g.step_raw(*args, hidden_in=h, check=False)
        assert rc == pkg.SHARD_EINVAL and "reset" in pkg.shard_last_error()
        # after a reset the step is correct again
        pkg.kv_state_reset(g.st, -1)
        prefill(g, TINY, SEED, 0, 40)
        o = OracleEngine(TINY, w, 1, 96)
        prefill(o, TINY, SEED, 0, 40)
        assert_close(g.step(*args, hidden_in=h), o.step(*args, hidden_in=h), what="after recovery")
        # and again, on the next step
        h2 = synth.hidden_in(TINY, SEED, 1, 1)
        args2 = ([1], np.array([41], np.int32), np.ones(42, np.uint8))
        assert_close(g.step(*args2, hidden_in=h2), o.step(*args2, hidden_in=h2), what="second step after recovery")
    finally:
        pkg.shard_debug_set_wait(sh.h, 1 << 22, -1)
        g.close()
        sh.close()
