"""The greedy speculative-decoding driver (paper_2608_19147_gb300.spec) on
the CPU: the acceptance rule, the rewind bookkeeping, and whole decodes over
the fp64 oracle (a tiny first+final stage and an oracle LM head), where
speculative decoding with mask-based rewind must emit exactly the tokens of
plain greedy decoding (Sections 5.2-5.4) -- and, the oracle being exact about
masked entries, the same top-1 probabilities bit for bit.  No GPU."""
import numpy as np
import pytest

import oracle
import synth
from paper_2608_19147_gb300.spec import GreedySpecDecoder, MaskedRequest, greedy_accept
from scenarios import OracleEngine

SHAPE = synth.TINY
SEED = 4242


def test_greedy_accept_rule():
    assert greedy_accept([], [7]) == (0, [7])
    assert greedy_accept([1, 2, 3], [1, 2, 3, 9]) == (3, [1, 2, 3, 9])
    assert greedy_accept([1, 5, 3], [1, 2, 3, 9]) == (1, [1, 2])
    assert greedy_accept([4, 2, 3], [1, 2, 3, 9]) == (0, [1])
    with pytest.raises(ValueError):
        greedy_accept([1, 2], [1, 2])


def test_masked_request_bookkeeping():
    r = MaskedRequest(3)
    pos, mask = r.inputs(3)
    assert pos.tolist() == [3, 4, 5] and mask.tolist() == [1] * 6
    r.commit(3, 1)   # two rejected drafts stay in the cache, masked
    pos, mask = r.inputs(2)
    assert pos.tolist() == [4, 5]           # logical positions continue after the kept entry
    assert mask.tolist() == [1, 1, 1, 1, 0, 0, 1, 1]
    assert r.physical == 6 and r.position == 4
    with pytest.raises(ValueError):
        r.commit(2, 3)


class OracleForward:
    """Tiny first+final stage on the oracle, with an oracle top-1 head."""

    def __init__(self, weights, head, capacity=160, round_points=True):
        self.eng = OracleEngine(SHAPE, weights, 1, capacity, round_points=round_points)
        self.head = head
        self.calls = 0

    def __call__(self, tokens, positions, mask):
        self.calls += 1
        out16 = self.eng.step([tokens.size], positions, mask, token_ids=tokens)
        tok, p, _, _ = oracle.head_top1(out16, self.head.norm, self.head.lm_head, self.head.rms_eps)
        self.last_p = p
        return tok


def _run(dec, fwd, n_tokens, drafts_for):
    """Decodes n_tokens; also returns the top-1 probability behind each
    emitted token (the outputs of the accepted prefix and the correction)."""
    out = [dec.prefill(drafts_for.prompt)]
    probs = [fwd.last_p[-1]]
    step = 0
    while len(out) < n_tokens:
        e = dec.step(drafts_for(out, step))
        probs += list(fwd.last_p[:len(e)])
        out += e
        step += 1
    return out[:n_tokens], np.array(probs[:n_tokens])


@pytest.fixture(scope="module")
def model():
    return synth.make_weights(SHAPE, SEED), synth.make_head(SHAPE.hidden, SHAPE.vocab, SHAPE.group, SEED + 1)


def _prompt(n):
    return synth.token_ids(SHAPE, SEED, 99, n).tolist()


class _NoDrafts:
    def __init__(self, prompt):
        self.prompt = prompt

    def __call__(self, out, step):
        return []


def _plain(model, n_tokens, prompt, with_probs=False):
    w, hw = model
    fwd = OracleForward(w, hw)
    out, probs = _run(GreedySpecDecoder(fwd), fwd, n_tokens, _NoDrafts(prompt))
    return (out, probs) if with_probs else out


def _drafts(truth, done, k, step, p=0.6):
    """Draft stand-in: the true continuation with probability p, else a
    seeded wrong token."""
    u = synth.uniform(k, seed=SEED, stream=500 + step, tag=synth.TAG_ACCEPT)
    wrong = synth.draft_tokens(SEED, step, k, SHAPE.vocab)
    d = []
    for j in range(k):
        good = truth[done + j] if done + j < len(truth) else int(wrong[j])
        d.append(good if u[j] < p else (int(wrong[j]) if int(wrong[j]) != good else (good + 1) % SHAPE.vocab))
    return d


@pytest.mark.parametrize("k", [2, 4])
def test_speculative_equals_plain_greedy_on_the_oracle(model, k):
    prompt = _prompt(21)   # two prefill blocks (16 + 5)
    truth, p_truth = _plain(model, 24, prompt, with_probs=True)
    w, hw = model
    fwd = OracleForward(w, hw)
    dec = GreedySpecDecoder(fwd)

    class Drafts(_NoDrafts):
        def __call__(self, out, step):
            return _drafts(truth, len(out), k, step)

    out, probs = _run(dec, fwd, len(truth), Drafts(prompt))
    assert out == truth
    assert np.array_equal(probs, p_truth)      # masked entries contribute nothing at all
    assert 0 < dec.accepted < dec.proposed      # some drafts accepted, some rewound
    assert dec.req.physical > dec.req.position  # rejected entries stay in the cache
    assert fwd.calls < 2 + len(truth)           # fewer forwards than plain decoding


def test_all_right_and_all_wrong_drafts(model):
    prompt = _prompt(9)
    truth = _plain(model, 13, prompt)
    w, hw = model
    dec = GreedySpecDecoder(OracleForward(w, hw))
    first = dec.prefill(prompt)
    assert first == truth[0]
    assert dec.step(truth[1:5]) == truth[1:6]          # all 4 accepted + the correction
    wrong = [(t + 1) % SHAPE.vocab for t in truth[6:10]]
    assert dec.step(wrong) == truth[6:7]               # none accepted: one token
    assert dec.req.valid[-4:] == [0, 0, 0, 0]


def test_unmasked_rejected_drafts_change_the_result(model):
    # teeth: a driver that kept rejected drafts visible computes something
    # else (this small random model's argmax barely depends on context, so
    # the probabilities show it)
    prompt = _prompt(4)
    truth, p_truth = _plain(model, 8, prompt, with_probs=True)
    w, hw = model
    fwd = OracleForward(w, hw)
    dec = GreedySpecDecoder(fwd)
    dec.prefill(prompt)
    wrong = synth.draft_tokens(SEED, 77, 15, SHAPE.vocab).tolist()
    assert dec.step(wrong) == truth[1:2]
    dec.req.valid = [1] * dec.req.physical             # forget the rewind
    probs = []
    for _ in range(6):
        dec.step([])
        probs.append(fwd.last_p[0])
    assert np.abs(np.array(probs) - p_truth[2:8]).max() > 1e-6
