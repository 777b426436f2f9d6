"""Host-side pins of the benchmark's workloads and of the bytes its roofline
divides by (no GPU).

- The algorithmic weight bytes per step of the 8B and 70B stages equal the
  figures worked out by hand from the Llama-3.1 shapes: 4 bits per code, an
  fp16 scale and a uint4 zero point per group of 128 inputs, every one of the
  seven matrices of every layer (Section 3.2 exports INT4 weights in groups
  of 128).
- Decode plans grow one cache entry per step with an all-ones mask and
  logical positions that follow the cache length.
- Verify plans follow the longest-prefix acceptance of greedy speculative
  decoding (Section 5.2): 1 + a of the 5 new entries become valid, the
  rejected drafts stay in the cache with mask 0 on every later step, and the
  logical position advances by 1 + a.  The stand-in draw of a (4 seeded
  Bernoulli(0.6), the count of leading successes) has the distribution that
  rule implies.
- Micro-batch plans apply a fresh uniform beam_idx permutation per step with
  gather-lineage semantics (Section 4: row b continues the sequence that row
  beam_idx[b] held).
- The KV term of the algorithmic bytes counts the entries attention must
  read (valid cache entries plus the new ones), never masked holes; the line
  also reports the physical count, holes included, and the cache bloat
  (physical over valid entries) that mask-based rewind costs.
"""
import numpy as np
import pytest

import bench
import synth

GB8_WEIGHT_BYTES = 1_812_987_904   # 3,489,660,928 weights: codes 1,744,830,464 + scales 54,525,952 + zeros 13,631,488
GB70_WEIGHT_BYTES = 8_890_613_760  # 17,112,760,320 weights: 8,556,380,160 + 267,386,880 + 66,846,720
KV_ENTRY_BYTES = 4096              # 8 kv heads x 128 dims x fp16 x (K, V), per layer


def test_weight_bytes_per_step_match_the_hand_worked_figures():
    assert bench.Plan("8b-decode", 1, bench.SEED).weight_bytes() == GB8_WEIGHT_BYTES
    assert bench.Plan("70b-decode", 1, bench.SEED).weight_bytes() == GB70_WEIGHT_BYTES
    # the 1.81 GB per step that no L2 flush is needed for: far above 129 MB
    assert GB8_WEIGHT_BYTES > 10 * 129e6


def test_kv_entry_bytes():
    assert synth.LLAMA8B_STAGE.kv_bytes_per_token() == KV_ENTRY_BYTES
    assert synth.LLAMA70B_STAGE.kv_bytes_per_token() == KV_ENTRY_BYTES
    assert synth.TINY.kv_bytes_per_token() == 512  # 2 kv heads x 64 dims x 2 B x 2


def test_decode_plan_grows_one_entry_per_step():
    K = 256
    p = bench.Plan("8b-decode", K, bench.SEED)
    s = p.shape
    io = 1 * s.hidden * 2 * 2
    norms = s.n_layers * 2 * s.hidden * 2
    for t, st in enumerate(p.steps):
        L = 72 + t
        assert st["beam"] is None
        assert st["pos"].tolist() == [L]
        assert st["mask"][0, :L + 1].all() and not st["mask"][0, L + 1:].any()
        assert st["tokens"].shape == (1,) and 0 <= int(st["tokens"][0]) < s.vocab
        assert p.alg_bytes(t) == GB8_WEIGHT_BYTES + (L + 1) * KV_ENTRY_BYTES * s.n_layers + io + norms
    # mean cache read of the 256-step request: entries 73..328, 200.5 on average
    mean_kv = np.mean([st["kv_bytes"] for st in p.steps])
    assert mean_kv == pytest.approx(200.5 * KV_ENTRY_BYTES * s.n_layers)
    # K steps beyond one request chain fresh requests from the same prefill
    p2 = bench.Plan("8b-decode", 300, bench.SEED)
    assert p2.R == 2 and p2.step_of[256] == (1, 0) and p2.steps[256]["pos"].tolist() == [72]


def test_verify_plan_masks_rejected_drafts_and_advances_by_accepted():
    K, n = 128, 5
    p = bench.Plan("8b-verify", K, bench.SEED)
    valid = [1] * 512
    pos = 512
    holes = 0
    for t, st in enumerate(p.steps):
        L = len(valid)
        assert L == 512 + n * t  # every step appends 5 entries; nothing is trimmed
        row = st["mask"][0]
        assert row[:L].tolist() == valid
        assert row[L:L + n].all() and not row[L + n:].any()
        assert st["pos"].tolist() == list(range(pos, pos + n))
        assert st["kv_bytes"] == (sum(valid) + n) * KV_ENTRY_BYTES * p.shape.n_layers
        a = synth.accepted_drafts(bench.SEED, t, n - 1)
        valid += [1] * (1 + a) + [0] * (n - 1 - a)
        pos += 1 + a
        holes += n - 1 - a
    assert len(valid) == 512 + n * K == 1152  # the physical cache length the workload reaches
    assert holes > 0  # masked holes accumulate mid-cache


def test_accepted_drafts_follow_longest_prefix_of_bernoulli():
    # a = number of leading successes of 4 Bernoulli(0.6) draws:
    # P(a = k) = 0.6^k 0.4 for k < 4, P(a = 4) = 0.6^4; E[a] = 1.3056
    n = 6000
    a = np.array([synth.accepted_drafts(7, t, 4) for t in range(n)])
    want = np.array([0.4, 0.24, 0.144, 0.0864, 0.1296])
    assert abs(a.mean() - 1.3056) < 4 * 1.4009 / np.sqrt(n)
    freq = np.bincount(a, minlength=5) / n
    assert np.all(np.abs(freq - want) < 4 * np.sqrt(want * (1 - want) / n)), freq
    # a draw of k drafts never accepts more than k
    assert max(synth.accepted_drafts(7, t, 2) for t in range(200)) <= 2


def test_microbatch_plan_applies_gather_lineage_each_step():
    K = 64
    p = bench.Plan("8b-microbatch", K, bench.SEED)
    lens = list(p.prefill[0])
    assert len(lens) == 8 and all(128 <= L <= 2048 for L in lens)
    perms = set()
    for t, st in enumerate(p.steps):
        beam = st["beam"]
        assert sorted(beam.tolist()) == list(range(8))
        perms.add(tuple(beam.tolist()))
        lens = [lens[j] for j in beam]  # row b continues the sequence of row beam[b]
        for b in range(8):
            assert st["mask"][b, :lens[b] + 1].all() and not st["mask"][b, lens[b] + 1:].any()
        assert st["pos"].tolist() == lens  # every entry is valid: position = length
        assert st["kv_bytes"] == sum(L + 1 for L in lens) * KV_ENTRY_BYTES * p.shape.n_layers
        lens = [L + 1 for L in lens]
    assert len(perms) > K // 2  # a fresh permutation per step


def test_beam_permutations_are_uniform():
    # Fisher-Yates over seeded uniforms: every element lands in every place
    # with probability 1/n, and a permutation has one fixed point on average
    # (a cyclic-only shuffle would have none)
    n, T = 8, 4000
    counts = np.zeros((n, n))
    fixed = 0
    for t in range(T):
        perm = synth.permutation(11, t, n)
        counts[np.arange(n), perm] += 1
        fixed += int(np.sum(perm == np.arange(n)))
    p = 1.0 / n
    assert np.all(np.abs(counts / T - p) < 5 * np.sqrt(p * (1 - p) / T)), counts
    assert abs(fixed / T - 1.0) < 0.1


def test_tiny_and_70b_plans():
    p = bench.Plan("tiny", 4, bench.SEED)
    assert p.M == 1 and p.steps[0]["pos"].tolist() == [72]
    p70 = bench.Plan("70b-verify", 3, bench.SEED)
    assert p70.M == 5 and p70.steps[0]["hidden"].shape == (5, 8192)
    assert p70.steps[0]["kv_bytes"] == (4096 + 5) * KV_ENTRY_BYTES * 20


def test_kv_counted_valid_and_physical_with_cache_bloat():
    # decode and micro-batch have no holes: both counts agree, no bloat
    for cfg, K in (("8b-decode", 256), ("8b-microbatch", 64)):
        k = bench.Plan(cfg, K, bench.SEED).kv_summary(K)
        assert k["valid_bytes_per_step"] == k["physical_bytes_per_step"]
        assert k["cache_bloat_mean"] == k["cache_bloat_last"] == 1.0
    # verify: every step appends 5 physical entries and 1 + a valid ones
    K = 128
    p = bench.Plan("8b-verify", K, bench.SEED)
    k = p.kv_summary(K)
    valid = 512 + sum(1 + synth.accepted_drafts(bench.SEED, t, 4) for t in range(K - 1))
    phys = 512 + 5 * (K - 1)
    assert k["cache_bloat_last"] == pytest.approx((phys + 5) / (valid + 5))
    assert k["physical_bytes_per_step"] > k["valid_bytes_per_step"]
    assert k["physical_bytes_per_step"] == pytest.approx(
        np.mean([512 + 5 * t + 5 for t in range(K)]) * KV_ENTRY_BYTES * 16)
    # the algorithmic bytes count valid entries only
    assert p.steps[3]["kv_bytes"] < p.steps[3]["kv_phys_bytes"]


def test_emitted_tokens_per_step():
    p = bench.Plan("8b-decode", 8, bench.SEED)
    assert all(st["emitted"] == 1 for st in p.steps)
    p = bench.Plan("8b-microbatch", 8, bench.SEED)
    assert all(st["emitted"] == 8 for st in p.steps)
    K = 128
    p = bench.Plan("8b-verify", K, bench.SEED)
    assert [st["emitted"] for st in p.steps] == [1 + synth.accepted_drafts(bench.SEED, t, 4) for t in range(K)]
