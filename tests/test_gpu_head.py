"""GPU parity of the final stage's LM head with the top-1 epilogue
(include/head.h, Section 6.7) and of greedy speculative decoding through it
(paper_2608_19147_gb300.spec, Sections 5.2-5.4), through the C ABI.

Logits: the GPU computes them in fp32 from the same fp16-rounded normalised
activations as the fp64 oracle; a normalised value can land one fp16 ulp
apart (fp32 vs fp64 norm), which moves a logit by at most |W| * 2^-11 * |x|,
so logits are compared within 2e-3 absolute plus 1e-4 relative to the
largest.  Tokens must agree wherever the oracle's top-2 margin exceeds 1e-2;
p_max within 1e-3 relative."""
import dataclasses

import numpy as np
import pytest
import torch

import oracle
import paper_2608_19147_gb300 as pkg
import synth
from gpu_engine import GpuShard, to_dev
from paper_2608_19147_gb300.spec import GreedySpecDecoder, ShardPipeline
from scenarios import OracleEngine

pytestmark = pytest.mark.gpu
SEED = 90210
MARGIN = 1e-2


class GpuHead:
    def __init__(self, hw):
        self.hw = hw
        self.h = pkg.head_create(hw.hidden, hw.vocab, hw.group, hw.rms_eps, hw.lm_head, hw.norm)

    def close(self):
        if self.h:
            pkg.head_destroy(self.h)
            self.h = None

    def run(self, h16):
        M = h16.shape[0]
        d_h = to_dev(h16)
        tok = torch.empty(M, dtype=torch.int32, device="cuda")
        p = torch.empty(M, dtype=torch.float32, device="cuda")
        ld = (self.hw.vocab + 3) // 4 * 4
        lg = torch.empty((M, ld), dtype=torch.float32, device="cuda")
        s = torch.cuda.current_stream().cuda_stream
        pkg.head_debug_logits(self.h, d_h.data_ptr(), M, lg.data_ptr(), ld, s)
        pkg.head_top1(self.h, d_h.data_ptr(), M, tok.data_ptr(), p.data_ptr(), s)
        torch.cuda.synchronize()
        return tok.cpu().numpy(), p.cpu().numpy(), lg.cpu().numpy()[:, :self.hw.vocab]


def _check_against_oracle(hw, h16, what):
    g = GpuHead(hw)
    try:
        tok, p, lg = g.run(h16)
        otok, op, omargin, olg = oracle.head_top1(h16, hw.norm, hw.lm_head, hw.rms_eps)
        scale = np.abs(olg).max()
        err = np.abs(lg - olg).max()
        assert err <= 2e-3 + 1e-4 * scale, "%s: logits max-abs %.3e (scale %.2f)" % (what, err, scale)
        sure = omargin > MARGIN
        assert sure.any(), what
        assert np.array_equal(tok[sure], otok[sure]), (what, tok, otok, omargin)
        assert np.allclose(p[sure], op[sure], rtol=1e-3, atol=0), (what, p, op)
        # the reported token is the argmax of the GPU's own logits, lowest id on ties
        assert np.array_equal(tok, lg.argmax(axis=1)), what
        return tok, p
    finally:
        g.close()


@pytest.mark.parametrize("M", [1, 5, 16])
def test_head_tiny_matches_oracle(M):
    hw = synth.make_head(256, 512, 32, SEED)
    _check_against_oracle(hw, synth.hidden_in(synth.TINY, SEED, M, M), "tiny M=%d" % M)


@pytest.mark.parametrize("V,H,group", [(1000, 320, 64), (777, 320, 32), (64, 128, 128), (3, 256, 128)])
def test_head_ragged_shapes_match_oracle(V, H, group):
    # vocab not a multiple of the 64-row block, hidden not a multiple of 128
    hw = synth.make_head(H, V, group, SEED + V)
    shape = dataclasses.replace(synth.TINY, hidden=H)
    _check_against_oracle(hw, synth.hidden_in(shape, SEED, 7, 4), "V=%d H=%d g=%d" % (V, H, group))


@pytest.mark.parametrize("M", [1, 3])
def test_head_llama8b_vocab_matches_oracle(M):
    # the Llama-3.1-8B final stage's head: 128256 x 4096, group 128
    hw = synth.make_head(4096, 128256, 128, SEED)
    _check_against_oracle(hw, synth.hidden_in(synth.LLAMA8B_STAGE, SEED, 11, M), "8B head M=%d" % M)


def test_head_host_entry_point_deterministic_and_rows_independent():
    hw = synth.make_head(256, 512, 32, SEED + 5)
    g = GpuHead(hw)
    try:
        h = synth.hidden_in(synth.TINY, SEED, 3, 16)
        t1, p1 = pkg.head_top1_host(g.h, h)
        t2, p2 = pkg.head_top1_host(g.h, h)
        assert np.array_equal(t1, t2) and np.array_equal(p1, p2)
        td, pd, _ = g.run(h)
        assert np.array_equal(t1, td) and np.array_equal(p1, pd)
        t5, p5 = pkg.head_top1_host(g.h, h[5:6])   # a row alone == the row in a batch
        assert t5[0] == t1[5] and p5[0] == p1[5]
    finally:
        g.close()


def test_head_errors():
    hw = synth.make_head(256, 512, 32, SEED)
    g = GpuHead(hw)
    try:
        d = to_dev(synth.hidden_in(synth.TINY, SEED, 0, 1))
        t = torch.empty(17, dtype=torch.int32, device="cuda")
        assert pkg.head_top1(g.h, d.data_ptr(), 0, t.data_ptr(), None, check=False) == pkg.SHARD_EINVAL
        assert pkg.head_top1(g.h, d.data_ptr(), 17, t.data_ptr(), None, check=False) == pkg.SHARD_EINVAL
        assert pkg.head_top1(g.h, 0, 1, t.data_ptr(), None, check=False) == pkg.SHARD_EINVAL
        assert "null" in pkg.shard_last_error()
        # still usable afterwards
        tok, p = pkg.head_top1_host(g.h, synth.hidden_in(synth.TINY, SEED, 0, 1))
        assert 0 <= tok[0] < 512 and 0 < p[0] <= 1
    finally:
        g.close()
    bad = dataclasses.replace(hw, group=48)
    with pytest.raises(pkg.ShardError) as e:
        pkg.head_create(bad.hidden, bad.vocab, 48, bad.rms_eps, bad.lm_head, bad.norm)
    assert e.value.code == pkg.SHARD_EUNSUPPORTED


# ---------------------------------------------------------------------------
# Greedy speculative decoding through shards and the head
# ---------------------------------------------------------------------------

def _oracle_pipeline(stages, head):
    """stages: [(shape, weights)], stage 0 with the embedding."""
    engs = [OracleEngine(s, w, 1, 192) for s, w in stages]

    def fwd(tokens, positions, mask):
        h = None
        for i, e in enumerate(engs):
            h = e.step([tokens.size], positions, mask, token_ids=tokens if i == 0 else None,
                       hidden_in=None if i == 0 else h)
        tok, p, margin, _ = oracle.head_top1(h, head.norm, head.lm_head, head.rms_eps)
        fwd.margins.append(margin)
        return tok

    fwd.margins = []
    return fwd


def _decode(fwd, prompt, n, drafts_for=None):
    dec = GreedySpecDecoder(fwd)
    out = [dec.prefill(prompt)]
    step = 0
    while len(out) < n:
        out += dec.step(drafts_for(out, step) if drafts_for else [])
        step += 1
    return out[:n], dec


def _split_stages():
    w = synth.make_weights(synth.TINY, SEED)
    s0 = dataclasses.replace(synth.TINY, name="tiny-stage0", n_layers=1)
    s1 = dataclasses.replace(synth.TINY, name="tiny-stage1", n_layers=1, vocab=0)
    w0 = synth.ShardWeights(s0, SEED, [w.layers[0]], w.embedding)
    w1 = synth.ShardWeights(s1, SEED, [w.layers[1]], None)
    return w, [(s0, w0), (s1, w1)]


def test_gpu_speculative_decoding_equals_plain_and_the_oracle():
    w, _ = _split_stages()
    head = synth.make_head(synth.TINY.hidden, synth.TINY.vocab, synth.TINY.group, SEED + 1)
    prompt = synth.token_ids(synth.TINY, SEED, 5, 19).tolist()
    n = 40
    # oracle plain greedy, with margins along the path
    ofwd = _oracle_pipeline([(synth.TINY, w)], head)
    truth, _ = _decode(ofwd, prompt, n)
    n_pre = -(-len(prompt) // pkg.SHARD_MAX_TOKENS)   # prefill blocks; the last one gives token 0
    margins = np.concatenate([m[-1:] for m in ofwd.margins[n_pre - 1:]])[:n]
    sure = n if (margins > MARGIN).all() else int(np.argmin(margins > MARGIN))
    assert sure >= 8, margins
    sh = GpuShard(synth.TINY, w)
    g = GpuHead(head)
    try:
        plain = ShardPipeline([sh.h], synth.TINY.hidden, g.h, 192)
        got, _ = _decode(plain, prompt, n)
        plain.close()
        assert got[:sure] == truth[:sure]

        def drafts(out, step, k=4):
            u = synth.uniform(k, seed=SEED, stream=900 + step, tag=synth.TAG_ACCEPT)
            wrong = synth.draft_tokens(SEED, 900 + step, k, synth.TINY.vocab)
            d = []
            for j in range(k):
                good = got[len(out) + j] if len(out) + j < n else int(wrong[j])
                d.append(good if u[j] < 0.6 else (int(wrong[j]) if int(wrong[j]) != good else (good + 1) % 512))
            return d

        spec = ShardPipeline([sh.h], synth.TINY.hidden, g.h, 192)
        out, dec = _decode(spec, prompt, n, drafts)
        spec.close()
        assert out == got                   # speculative == plain greedy on the GPU
        assert 0 < dec.accepted < dec.proposed
    finally:
        g.close()
        sh.close()


def test_gpu_two_stage_pipeline_matches_the_oracle_pipeline():
    # the tiny model split into two one-layer stages; the fp16 hidden states
    # cross from stage to stage as in the paper's relay (Section 3.3)
    _, stages = _split_stages()
    head = synth.make_head(synth.TINY.hidden, synth.TINY.vocab, synth.TINY.group, SEED + 1)
    prompt = synth.token_ids(synth.TINY, SEED, 6, 12).tolist()
    n = 24
    ofwd = _oracle_pipeline(stages, head)
    truth, _ = _decode(ofwd, prompt, n)
    n_pre = -(-len(prompt) // pkg.SHARD_MAX_TOKENS)   # prefill blocks; the last one gives token 0
    margins = np.concatenate([m[-1:] for m in ofwd.margins[n_pre - 1:]])[:n]
    sure = n if (margins > MARGIN).all() else int(np.argmin(margins > MARGIN))
    assert sure >= 6, margins
    shards = [GpuShard(s, sw) for s, sw in stages]
    g = GpuHead(head)
    try:
        pipe = ShardPipeline([s.h for s in shards], synth.TINY.hidden, g.h, 192)
        got, _ = _decode(pipe, prompt, n)
        pipe.close()
        assert got[:sure] == truth[:sure]
    finally:
        g.close()
        for s in shards:
            s.close()
