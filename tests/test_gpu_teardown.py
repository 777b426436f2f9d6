"""A shard_create that fails part-way frees what it had allocated.

A null norm vector in a layer is found only after the layer's weights were
uploaded and repacked, so the call has by then allocated the weight pool
(113 MB for one 8B-shaped layer) and its staging.  It must return EINVAL and
leave the device's free memory where it was: a caller that retries, or that
creates a smaller shard instead, must not find HBM held by a shard that never
existed.
"""
import dataclasses

import pytest
import torch

import paper_2608_19147_gb300 as pkg
import synth

pytestmark = pytest.mark.gpu


def test_failed_create_frees_its_device_buffers():
    shape = dataclasses.replace(synth.LLAMA8B_STAGE, name="8b-1layer", n_layers=1, vocab=0)
    w = synth.make_weights(shape, 2)
    cfg = pkg.make_config(shape)
    # a complete create and destroy first: the library's kernels are loaded
    # once, and their code stays resident
    pkg.shard_destroy(pkg.shard_create(cfg, w.layers, w.embedding))
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    bad = [dataclasses.replace(w.layers[0], ffn_norm=None)]
    for _ in range(3):
        with pytest.raises(pkg.ShardError) as e:
            pkg.shard_create(cfg, bad, w.embedding)
        assert e.value.code == pkg.SHARD_EINVAL and "null norm" in str(e.value)
    torch.cuda.synchronize()
    free1 = torch.cuda.mem_get_info()[0]
    assert free0 - free1 < (32 << 20), "failed creates kept %.1f MB" % ((free0 - free1) / 1e6)
    # and a complete shard can still be created afterwards
    h = pkg.shard_create(cfg, w.layers, w.embedding)
    pkg.shard_destroy(h)
