#!/usr/bin/env python
"""Benchmark of the GB300 shard-decode path.

Metric: INT4 shard decode tokens/s at 1 GB300, with the achieved HBM
bandwidth of the step kernel (the whole decode step is one launch) against
the measured peak.

Default workload (the Llama-3.1-8B-shaped stage 1 of 2 decode): a 16-layer
shard (hidden 4096, 32 q / 8 kv heads, head_dim 128, FFN 14336, uint4 group
128), token ids looked up in the shard's 128256 x 4096 embedding, one request
with a 72-token fp16 cache decoding one token per step for 256 steps,
identity beam_idx, all-ones attention_mask.  A run of K steps chains
ceil(K / 256) such requests back to back (each from its own 72-token cache),
so every step is a step of that workload.  Weights are seeded synthetic
(no checkpoints are available); the 1.81 GB of packed weights per step are
far larger than L2, so no L2 flush is needed between steps.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl gb300|reference]
                  [--config 8b-decode|8b-verify|8b-microbatch|70b-decode|70b-verify|tiny|8b-head|8b-head-verify|8b-prefill]
                  [--no-cpu-baseline] [--no-other-workloads] [--layers N]

At one GPU the default (8b-decode) line also carries `other_workloads`: the
8B verify and micro-batch and the 70B decode and verify workloads, each run
afterwards as `bench.py --config <name>` in a child process of its own, with
its value, step time and roofline fraction.

Under torchrun each rank runs an independent replica on its own GPU
(replicas only: the path has no exchange step) and rank 0 prints one JSON
line.
"""
from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402

METRIC = "INT4 shard decode tokens/s at 1 GB300; achieved HBM GB/s vs ~8 TB/s peak"
SEED = 20260802
CONFIGS = {
    "8b-decode": dict(shape=synth.LLAMA8B_STAGE, prefill=72, steps_per_request=256, rows=1, n=1, tokens=True,
                      workload="llama3.1-8b-stage1of2 16L decode: 1 request, 72-token prefill, 1 token/step, "
                               "256 steps per request, identity beam_idx, all-ones mask"),
    "8b-verify": dict(shape=synth.LLAMA8B_STAGE, prefill=512, steps_per_request=128, rows=1, n=5, tokens=False,
                      workload="llama3.1-8b-stage1of2 16L speculative verify: 1 request, 512-token prefill, "
                               "1+4 rows/step, Bernoulli(0.6) prefix accept, rejected rows masked, 128 steps"),
    "8b-microbatch": dict(shape=synth.LLAMA8B_STAGE, prefill=None, steps_per_request=64, rows=8, n=1, tokens=False,
                          workload="llama3.1-8b-stage1of2 16L micro-batch: 8 requests, lengths U{128..2048}, "
                                   "random beam_idx permutation per step, 1 token/request/step, 64 steps"),
    "70b-decode": dict(shape=synth.LLAMA70B_STAGE, prefill=4096, steps_per_request=64, rows=1, n=1, tokens=False,
                       workload="llama3.1-70b-stage1of4 20L decode: 1 request, 4096-token prefill, 1 token/step, "
                                "64 steps"),
    "70b-verify": dict(shape=synth.LLAMA70B_STAGE, prefill=4096, steps_per_request=64, rows=1, n=5, tokens=False,
                       workload="llama3.1-70b-stage1of4 20L speculative verify: 4096-token prefill, 1+4 rows/step, "
                                "Bernoulli(0.6) prefix accept, 64 steps"),
    "tiny": dict(shape=synth.TINY, prefill=72, steps_per_request=256, rows=1, n=1, tokens=True,
                 workload="tiny 2L h256 decode: 72-token prefill, 1 token/step"),
    # the final stage's LM head with top-1 compression (Section 6.7), not a shard step
    "8b-head": dict(head=(4096, 128256, 128), rows=1,
                    workload="llama3.1-8b final-stage LM head, top-1: RMSNorm + 128256x4096 INT4 lm_head + "
                             "argmax/p_max, 1 hidden row per call"),
    "8b-head-verify": dict(head=(4096, 128256, 128), rows=5,
                           workload="llama3.1-8b final-stage LM head, top-1: RMSNorm + 128256x4096 INT4 lm_head + "
                                    "argmax/p_max, 1+4 verify rows per call"),
    # prefill of a prompt through the stage (Section 3.4), projections on the tensor cores
    "8b-prefill": dict(prefill_tokens=512, shape=synth.LLAMA8B_STAGE, rows=512,
                       workload="llama3.1-8b-stage1of2 16L prefill: one 512-token prompt (token ids) onto an empty "
                                "row per call, chunks of 256 tokens, projections as tcgen05 GEMMs"),
}
HEAD_METRIC = "LM-head top-1 rows/s at 1 GB300 (final stage, Section 6.7); achieved HBM GB/s"
PREFILL_METRIC = "INT4 shard prefill tokens/s at 1 GB300; achieved tensor TFLOP/s of the projections"


def log(*a):
    print(*a, file=sys.stderr, flush=True)


# ---------------------------------------------------------------------------
# Workload: per-step inputs (host), built from the seeded generator
# ---------------------------------------------------------------------------

class Plan:
    """Host-side step plan of one workload: for each step, n_new per row,
    position ids, the attention mask rows, beam_idx and token ids or hidden
    states; per-row prefill lengths; the byte counts of the step."""

    def __init__(self, cfg_name: str, K: int, seed: int, request0: int = 0, shape=None):
        c = CONFIGS[cfg_name]
        self.name, self.c, self.shape = cfg_name, c, (shape or c["shape"])
        s = self.shape
        self.B = c["rows"]
        self.n = c["n"]
        self.M = self.B * self.n
        self.spr = c["steps_per_request"]
        self.K = K
        self.R = max(1, -(-K // self.spr))  # requests (each with its own cache)
        if c["prefill"] is None:
            self.prefill = [synth.lengths(seed + request0 + r, self.B, 128, 2048).tolist() for r in range(self.R)]
        else:
            self.prefill = [[c["prefill"]] * self.B for _ in range(self.R)]
        self.cap = max(max(p) for p in self.prefill) + self.spr * self.n + 8
        self.stride = self.cap
        self.steps = []
        for r in range(self.R):
            lens = list(self.prefill[r])     # logical (cache) length per row
            valid = [[1] * L for L in lens]  # live entries per row
            pos = list(lens)                 # logical positions
            for j in range(self.spr):
                t = r * self.spr + j
                if t >= K:
                    break
                beam = None
                if cfg_name == "8b-microbatch":
                    beam = synth.permutation(seed, t, self.B)
                    lens = [lens[p] for p in beam]
                    valid = [list(valid[p]) for p in beam]
                    pos = [pos[p] for p in beam]
                mask = np.zeros((self.B, self.stride), np.uint8)
                positions = []
                for b in range(self.B):
                    L = lens[b]
                    mask[b, :L] = np.array(valid[b], np.uint8)
                    mask[b, L:L + self.n] = 1
                    positions += list(range(pos[b], pos[b] + self.n))
                step = dict(mask=mask, pos=np.array(positions, np.int32), beam=beam)
                if c["tokens"]:
                    step["tokens"] = synth.token_ids(s, seed, t, self.M)
                else:
                    step["hidden"] = synth.hidden_in(s, seed, t, self.M)
                kv_read = kv_phys = 0
                for b in range(self.B):
                    # K and V of the entries attention must read: the live
                    # cache entries and the new ones, in every layer
                    kv_read += (sum(valid[b]) + self.n) * s.kv_bytes_per_token() * s.n_layers
                    # and of every physical entry, masked holes included
                    kv_phys += (lens[b] + self.n) * s.kv_bytes_per_token() * s.n_layers
                step["kv_bytes"] = kv_read
                step["kv_phys_bytes"] = kv_phys
                step["entries"] = (sum(lens) + self.B * self.n, sum(sum(v) for v in valid) + self.B * self.n)
                self.steps.append(step)
                acc = self.n
                if self.n > 1:
                    acc = 1 + synth.accepted_drafts(seed, t, self.n - 1)
                step["emitted"] = acc * self.B  # tokens the step emits: the accepted drafts and the correction
                for b in range(self.B):
                    valid[b] += [1] * acc + [0] * (self.n - acc)
                    lens[b] += self.n
                    pos[b] += acc
        self.step_of = [(t // self.spr, t % self.spr) for t in range(K)]

    def weight_bytes(self) -> int:
        return self.shape.packed_bytes_per_layer() * self.shape.n_layers

    def alg_bytes(self, t: int) -> int:
        """Algorithmic HBM bytes of step t: packed weights + scales + zeros,
        K/V of the entries attention reads, embedding rows or hidden states in,
        hidden states out, norm weights."""
        s = self.shape
        io = self.M * s.hidden * 2 * 2
        norms = s.n_layers * 2 * s.hidden * 2
        return self.weight_bytes() + self.steps[t]["kv_bytes"] + io + norms

    def kv_summary(self, K: int) -> dict:
        """KV read per step counted twice (valid entries, as in the
        algorithmic bytes, and physical entries including masked holes), and
        the cache bloat: the step's physical entries over its valid ones
        (cache plus new entries), mean over the steps and at the last step."""
        st = self.steps[:K]
        ratios = [phys / val for phys, val in (x["entries"] for x in st)]
        return {"valid_bytes_per_step": sum(x["kv_bytes"] for x in st) / K,
                "physical_bytes_per_step": sum(x["kv_phys_bytes"] for x in st) / K,
                "cache_bloat_mean": sum(ratios) / K, "cache_bloat_last": ratios[-1]}

    def kind_bytes(self, kind: str) -> int:
        """Algorithmic bytes of one launch of a projection kind."""
        s = self.shape
        names = {"qkv": ("q", "k", "v"), "o": ("o",), "gate_up": ("gate", "up"), "down": ("down",)}[kind]
        total = 0
        for nme in names:
            r, c = s.matrix_shape(nme)
            G = -(-c // s.group)
            total += r * c // 2 + r * G * 2 + r * G // 2 + self.M * c * 2 + self.M * r * 2
        return total


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.samples = []
        self.proc = None
        try:
            cmd = ["nvidia-smi", "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits", "-lms", "100"]
            if gpu_id:
                cmd += ["-i", gpu_id]
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception as e:  # no nvidia-smi
            log("clock sampling unavailable:", e)

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) >= 9:
                self.samples.append((time.time(), parts))

    def stop(self):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self, t0: float, t1: float):
        win = [p for (ts, p) in self.samples if t0 <= ts <= t1]
        if len(win) < 3:  # short timed region: widen to the samples next to it
            mid = 0.5 * (t0 + t1)
            win = [p for (ts, p) in sorted(self.samples, key=lambda x: abs(x[0] - mid))[:5]]
        if not win:
            return None

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None

        sm = [num(p[1]) for p in win if num(p[1]) is not None]
        mx = [num(p[2]) for p in win if num(p[2]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for p in win for i in range(4) if p[5 + i].lower().startswith("active")})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(win)}


def max_over_ranks(x: float, dist, device) -> float:
    """The largest of every rank's value (the slowest replica's time); x
    itself on a single process."""
    if dist is None:
        return x
    import torch

    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_throughput(world: int, units_per_rank: float, seconds: float) -> float:
    """Whole-job throughput of `world` independent replicas that each
    processed units_per_rank units, timed by the slowest one."""
    return world * units_per_rank / seconds


def measured_peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        return {}


KERNEL_SOURCES = {
    "step": ("gemv_core.cuh", "step_kernel.cu", "common.cuh", "kernels.h"),
    "head": ("gemv_core.cuh", "gemv.cu", "head.cu", "common.cuh", "kernels.h"),
}


def kernel_source_hash(kind: str = "step") -> str:
    h = hashlib.sha256()
    for f in KERNEL_SOURCES[kind]:
        h.update(open(os.path.join(ROOT, "paper_2608_19147_gb300", "csrc", f), "rb").read())
    return h.hexdigest()[:16]


def profiled_traffic(kind: str, cfg: str):
    """DRAM bytes per launch from a committed ncu summary, if it was taken on
    the current kernel source."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        data = json.load(open(path))
        ent = data.get("%s/%s" % (cfg, kind))
        if ent and ent.get("kernel_hash") == kernel_source_hash(kind):
            return ent.get("dram_bytes_per_launch")
    except Exception:
        pass
    return None


def stage_shape(args):
    """The configuration's stage, or its first --layers layers (a shallower
    slice of the same kernel, used for profiling captures)."""
    shape = CONFIGS[args.config]["shape"]
    if args.layers and args.layers != shape.n_layers:
        shape = dataclasses.replace(shape, name="%s-first%dL" % (shape.name, args.layers), n_layers=args.layers)
    return shape


def run_gpu(args, rank: int, world: int):
    import torch

    import paper_2608_19147_gb300 as pkg

    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", "0")))
    torch.cuda.set_device(dev)
    dist = None
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl", device_id=dev)
    c = CONFIGS[args.config]
    shape = stage_shape(args)
    K, W = args.steps, max(3, args.warmup)
    threads = max(1, (os.cpu_count() or 1) // max(1, int(os.environ.get("LOCAL_WORLD_SIZE", world))))
    t_gen = time.time()
    weights = synth.make_weights(shape, SEED, threads=threads)
    log("weights generated in %.1fs (%.2f GB packed)" % (time.time() - t_gen, weights.packed_bytes() / 1e9))
    plan = Plan(args.config, K, SEED, shape=shape)
    warm = Plan(args.config, W, SEED + 1, shape=shape)
    sh = pkg.shard_create(pkg.make_config(shape), weights.layers, weights.embedding)
    stream = torch.cuda.current_stream(dev)
    sptr = stream.cuda_stream

    def load_states(p: Plan):
        sts = []
        for r in range(p.R):
            st = pkg.kv_state_alloc(sh, p.B, p.cap)
            for b in range(p.B):
                for layer in range(shape.n_layers):
                    k, v = synth.kv_prefill(shape, SEED + r, b, p.prefill[r][b], layer)
                    pkg.kv_state_load(st, b, layer, k, v)
            sts.append(st)
        return sts

    def stage(p: Plan):
        """Per-step inputs resident on the device before timing."""
        to = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
        d = dict(mask=to(np.stack([s["mask"] for s in p.steps])), pos=to(np.stack([s["pos"] for s in p.steps])))
        if c["tokens"]:
            d["tok"] = to(np.stack([s["tokens"] for s in p.steps]))
        else:
            d["hid"] = to(np.stack([s["hidden"] for s in p.steps]).view(np.int16))
        if p.steps[0]["beam"] is not None:
            d["beam"] = to(np.stack([s["beam"] for s in p.steps]))
        d["out"] = torch.empty((p.M, shape.hidden), dtype=torch.int16, device=dev)
        return d

    def run_steps(p: Plan, sts, d, count):
        n_new = [p.n] * p.B

        def ptrs(key):  # device address of step t's slice, precomputed
            if key not in d:
                return [None] * count
            a = d[key]
            return [a.data_ptr() + t * a.stride(0) * a.element_size() for t in range(count)]

        tok, hid, beam, pos, mask = ptrs("tok"), ptrs("hid"), ptrs("beam"), ptrs("pos"), ptrs("mask")
        out = d["out"].data_ptr()
        state_of = [sts[p.step_of[t][0]] for t in range(count)]
        for t in range(count):
            pkg.shard_step(sh, state_of[t], hid[t], tok[t], n_new, pos[t], mask[t], p.stride, beam[t], out, sptr)

    def run_steps_one(p: Plan, sts, d, t):
        r, _ = p.step_of[t]
        g = lambda key: (d[key][t].data_ptr() if key in d else None)
        pkg.shard_step(sh, sts[r], g("hid"), g("tok"), [p.n] * p.B, d["pos"][t].data_ptr(), d["mask"][t].data_ptr(),
                       p.stride, g("beam"), d["out"].data_ptr(), sptr)

    # warm-up (own states, so the timed requests start from their prefills)
    wst, wd = load_states(warm), stage(warm)
    run_steps(warm, wst, wd, W)
    torch.cuda.synchronize()
    pkg.shard_sync_status(sh, sptr)
    sts, d = load_states(plan), stage(plan)
    gpu_id = ""
    try:
        gpu_id = str(torch.cuda.get_device_properties(dev).uuid)
        if gpu_id and not gpu_id.startswith("GPU-"):
            gpu_id = "GPU-" + gpu_id
    except Exception:
        gpu_id = ""
    sampler = ClockSampler(gpu_id)
    time.sleep(0.3)
    # ---- timed region ----
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    w0 = time.time()
    e0.record(stream)
    run_steps(plan, sts, d, K)
    e1.record(stream)
    torch.cuda.synchronize()
    w1 = time.time()
    if dist:
        dist.barrier()
    ms = e0.elapsed_time(e1)
    sampler.stop()
    clocks = sampler.summary(w0, w1)
    pkg.shard_sync_status(sh, sptr)
    ms = max_over_ranks(ms, dist, dev)
    for st in sts + wst:
        pkg.kv_state_free(st)

    # ---- per-phase times: the step kernel's barrier timestamps, averaged
    # over a pass of the same workload (one step, then read, per step) ----
    prof_K = min(K, 64)
    pplan = Plan(args.config, prof_K, SEED + 2, shape=shape)
    pst, pd = load_states(pplan), stage(pplan)
    PHASES = list(pkg.PHASES)
    n_ph = len(PHASES) * shape.n_layers + 1
    acc = np.zeros(n_ph)
    for t in range(prof_K):
        run_steps_one(pplan, pst, pd, t)
        acc += np.array(pkg.shard_debug_phase_times(sh, shape.n_layers))
    acc /= prof_K
    # times[0]: the prologue with the first RMSNorm and q|k|v projection;
    # then per layer: attention (after the first layer, with that layer's
    # RMSNorm and q|k|v projection in front), o, RMSNorm + gate|up, down
    phases = {"prologue_norm_qkv0": {"total_us_per_step": float(acc[0])}}
    lay = acc[1:].tolist()
    for i, name in enumerate(PHASES):
        v = np.array(lay[i::len(PHASES)])
        phases[name] = {"avg_us_per_layer": float(v.mean()), "total_us_per_step": float(v.sum())}
    for name, kind in (("o", "o"), ("gate_up", "gate_up"), ("down", "down")):
        t_us = phases[name]["avg_us_per_layer"]
        if t_us > 0:
            phases[name]["achieved_gbs"] = pplan.kind_bytes(kind) / (t_us * 1e3)
    for st in pst:
        pkg.kv_state_free(st)

    # ---- end to end through the host-buffer entry point ----
    eplan = Plan(args.config, K, SEED + 3, shape=shape)
    est = load_states(eplan)
    out = np.empty((eplan.M, shape.hidden), np.uint16)
    h2d = d2h = 0
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    t0 = time.perf_counter()
    for t in range(K):
        r, _ = eplan.step_of[t]
        s = eplan.steps[t]
        pkg.shard_step_host(sh, est[r], s.get("hidden"), s.get("tokens"), [eplan.n] * eplan.B, s["pos"], s["mask"],
                            s["beam"], out, sptr)
    t1 = time.perf_counter()
    s0 = eplan.steps[0]
    h2d = (s0["mask"].nbytes + s0["pos"].nbytes + (s0["tokens"].nbytes if "tokens" in s0 else s0["hidden"].nbytes)
           + (s0["beam"].nbytes if s0["beam"] is not None else 0))
    d2h = out.nbytes
    e2e_s = t1 - t0
    e2e_s = max_over_ranks(e2e_s, dist, dev)
    for st in est:
        pkg.kv_state_free(st)
    pkg.shard_destroy(sh)

    if rank != 0:
        if dist:
            dist.destroy_process_group()
        return
    peaks = measured_peaks()
    peak = peaks.get("hbm_gbs")
    peak_note = "of measured" if peak else "of fallback"
    if not peak:
        peak = 6800.0
    rows_per_step = plan.M
    value = replica_throughput(world, K * rows_per_step, ms / 1e3)
    step_bytes = sum(plan.alg_bytes(t) for t in range(K)) / K
    launches_per_step = 1  # the whole step is one kernel
    result = {
        "metric": METRIC,
        "value": value,
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": K,
        "warmup": W,
        "ms_per_step": ms / K,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "w4a16 (uint4 weights, fp16 activations, fp32 accumulate)",
        "data": "synthetic (seeded Gaussian weights quantised to uint4; no checkpoints available)",
        "config": {
            "workload": c["workload"] + ("" if shape.n_layers == c["shape"].n_layers else
                                         " [profiling slice: first %d layers only]" % shape.n_layers),
            "shard": "%s: %d layers, hidden %d, %dq/%dkv heads, head_dim %d, ffn %d, group %d" % (
                shape.name, shape.n_layers, shape.hidden, shape.n_heads, shape.n_kv_heads, shape.head_dim, shape.ffn,
                shape.group),
            "rows_per_step": rows_per_step,
            "requests_chained": plan.R,
            "l2": "no flush: each step streams %.2f GB of packed weights, far larger than the 129 MB L2" % (
                plan.weight_bytes() / 1e9),
            "inputs": "value: every step's inputs (token ids or hidden rows, positions, mask rows, beam_idx) are "
                      "resident in HBM before the timed region, which holds only the step launches; e2e times "
                      "the same steps through shard_step_host with each step's uploads and the output read-back",
            "parallelism": "replicas" if world > 1 else "single GPU",
            "seed": SEED,
        },
        "step_alg_bytes": step_bytes,
        "kv": plan.kv_summary(K),
        # a verify step processes 1 + 4 rows but emits 1 + accepted tokens
        "emitted_tokens_per_s": replica_throughput(world, sum(plan.steps[t]["emitted"] for t in range(K)), ms / 1e3),
        "roofline": {
            "kernel": "step_kernel (the whole decode step: %d layers in one launch)" % shape.n_layers,
            "bound": "hbm",
            "achieved": step_bytes / (ms / K * 1e6),
            "peak": peak,
            "unit": "GB/s",
            "frac": step_bytes / (ms / K * 1e6) / peak,
            "peak_note": "%s: MEASURED_PEAKS.json hbm_gbs (a copy bandwidth); achieved = algorithmic bytes per "
                         "launch / CUDA-event time of the timed launches" % peak_note,
            "traffic": profiled_traffic("step", args.config) if shape.n_layers == c["shape"].n_layers else None,
            "frac_of_8tbs_nominal": step_bytes / (ms / K * 1e6) / 8000.0,
        },
        "phases": phases,
        "e2e": {"value": replica_throughput(world, K * rows_per_step, e2e_s), "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h},
        "gpu_launches": K * launches_per_step,
        "clocks": clocks,
    }
    if want_other_workloads(args, world):
        log("measuring the other step workloads in child processes")
        result["other_workloads"] = other_workloads()
    if world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = cpu_baseline(args.config, weights, budget_s=args.cpu_budget)
    print(json.dumps(result), flush=True)
    if dist:
        dist.destroy_process_group()


# The other step workloads, measured by this script in child processes after
# the main line's timed region, so that one default run reports every shard
# workload; each child is `bench.py --config <name>` with its own timing.
OTHER_WORKLOADS = (("70b-decode", 64), ("8b-verify", 128), ("8b-microbatch", 64), ("70b-verify", 64))
LAUNCHER_ENV = ("RANK", "WORLD_SIZE", "LOCAL_RANK", "LOCAL_WORLD_SIZE", "GROUP_RANK", "ROLE_RANK", "ROLE_WORLD_SIZE",
                "GROUP_WORLD_SIZE", "MASTER_ADDR", "MASTER_PORT")


def want_other_workloads(args, world: int) -> bool:
    return (world == 1 and args.config == "8b-decode" and args.layers == 0 and not args.no_cpu_baseline
            and not args.no_other_workloads)


def _child_cmd(cfg: str, steps: int):
    return [sys.executable, os.path.abspath(__file__), "--config", cfg, "--steps", str(steps), "--warmup", "3",
            "--no-cpu-baseline"]


def _child_env():
    return {k: v for k, v in os.environ.items() if k not in LAUNCHER_ENV and not k.startswith("TORCHELASTIC_")}


def other_workloads(timeout_s: float = 150.0, total_s: float = 400.0) -> dict:
    """Runs each of OTHER_WORKLOADS in a child process of its own and returns
    its headline figures (or the reason it gave none): a child that fails
    cannot disturb the main line, which is complete before they start.  Each
    child gets timeout_s, all of them together total_s (each took under 30 s
    on a GB300); children that would start past that are skipped."""
    out = {}
    start = time.time()
    for cfg, steps in OTHER_WORKLOADS:
        t0 = time.time()
        left = total_s - (t0 - start)
        if left < 10.0:
            out[cfg] = {"error": "skipped: the other workloads' %.0f s were spent" % total_s}
            continue
        try:
            r = subprocess.run(_child_cmd(cfg, steps), capture_output=True, text=True, timeout=min(timeout_s, left),
                               env=_child_env())
            lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
            if r.returncode != 0 or not lines:
                tail = (r.stderr.strip().splitlines() or ["no output"])[-1]
                out[cfg] = {"error": "exit %d: %s" % (r.returncode, tail[:300])}
                continue
            d = json.loads(lines[-1])
            rf = d["roofline"]
            out[cfg] = {"workload": d["config"]["workload"], "value": d["value"], "unit": d["unit"],
                        "ms_per_step": d["ms_per_step"], "steps": d["steps"], "achieved_gbs": rf["achieved"],
                        "frac": rf["frac"], "peak": rf["peak"], "e2e": d["e2e"]["value"], "clocks": d["clocks"],
                        "gpu_launches": d["gpu_launches"], "kv": d.get("kv"),
                        "emitted_tokens_per_s": d.get("emitted_tokens_per_s"), "wall_s": round(time.time() - t0, 1)}
        except Exception as e:  # timeout, unparsable output
            out[cfg] = {"error": "%s: %s" % (type(e).__name__, str(e)[:300])}
    return out


# ---------------------------------------------------------------------------
# CPU oracle arm
# ---------------------------------------------------------------------------

def cpu_baseline(cfg_name: str, weights, budget_s: float = 20.0, max_steps: int = 256, one_thread: bool = True):
    """The fp64 CPU oracle, as it stands, on a bounded sample of the workload:
    the first steps of one request, until about budget_s seconds of work."""
    import oracle

    threads = os.cpu_count() or 1
    oracle.set_threads(threads)
    plan = Plan(cfg_name, max_steps, SEED)
    shape = plan.shape
    ref = oracle.OracleShard(shape, weights)
    st = ref.state(plan.B, plan.cap)
    for b in range(plan.B):
        for layer in range(shape.n_layers):
            k, v = synth.kv_prefill(shape, SEED + 0, b, plan.prefill[0][b], layer)
            st.load(b, layer, k, v)
    n = 0
    t0 = time.perf_counter()
    while n < min(max_steps, plan.spr):
        s = plan.steps[n]
        rc, _, _ = st.step([plan.n] * plan.B, s["pos"], s["mask"], hidden_in=s.get("hidden"),
                           token_ids=s.get("tokens"), beam_idx=s["beam"])
        assert rc == 0, rc
        n += 1
        if time.perf_counter() - t0 > budget_s:
            break
    el = time.perf_counter() - t0
    out = {"value": n * plan.M / el, "unit": "tokens/s", "cores": threads, "kind": "oracle",
           "sample": "first %d steps of one request of the %s workload (%d rows/step), fp64 oracle, "
                     "OpenMP over output rows with %d threads, %.1f s" % (n, cfg_name, plan.M, threads, el)}
    # the same oracle on one thread: the next steps of the request, when one
    # step fits in the budget
    est = el / max(n, 1) * threads
    if one_thread and threads > 1 and n < min(max_steps, plan.spr) and est <= 1.5 * budget_s:
        oracle.set_threads(1)
        n1 = 0
        t1 = time.perf_counter()
        while n + n1 < min(max_steps, plan.spr):
            s = plan.steps[n + n1]
            rc, _, _ = st.step([plan.n] * plan.B, s["pos"], s["mask"], hidden_in=s.get("hidden"),
                               token_ids=s.get("tokens"), beam_idx=s["beam"])
            assert rc == 0, rc
            n1 += 1
            if time.perf_counter() - t1 > budget_s / 2:
                break
        el1 = time.perf_counter() - t1
        oracle.set_threads(threads)
        out["value_1_thread"] = n1 * plan.M / el1
        out["sample_1_thread"] = "the next %d steps on 1 thread, %.1f s" % (n1, el1)
    return out


def head_cpu_baseline(hw, M: int, budget_s: float = 20.0):
    """The fp64 oracle head on a bounded sample: calls of M seeded rows until
    about budget_s seconds of work."""
    import oracle

    threads = os.cpu_count() or 1
    oracle.set_threads(threads)
    shape = dataclasses.replace(synth.LLAMA8B_STAGE, hidden=hw.hidden)
    n = 0
    t0 = time.perf_counter()
    while True:
        oracle.head_top1(synth.hidden_in(shape, SEED, 10000 + n, M), hw.norm, hw.lm_head, hw.rms_eps)
        n += 1
        if time.perf_counter() - t0 > budget_s:
            break
    el = time.perf_counter() - t0
    return {"value": n * M / el, "unit": "rows/s", "cores": threads, "kind": "oracle",
            "sample": "%d calls of %d rows of the LM-head workload, fp64 oracle, OpenMP over vocabulary rows with "
                      "%d threads, %.1f s" % (n, M, threads, el)}


def run_head(args, rank: int, world: int):
    """LM head with the top-1 epilogue: K calls of head_top1 on resident
    hidden rows, CUDA-event timed; e2e through head_top1_host."""
    import torch

    import paper_2608_19147_gb300 as pkg

    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", "0")))
    torch.cuda.set_device(dev)
    dist = None
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl", device_id=dev)
    c = CONFIGS[args.config]
    H, V, g = c["head"]
    M = c["rows"]
    K, W = args.steps, max(3, args.warmup)
    hw = synth.make_head(H, V, g, SEED)
    head = pkg.head_create(H, V, g, hw.rms_eps, hw.lm_head, hw.norm)
    stream = torch.cuda.current_stream(dev)
    sptr = stream.cuda_stream
    shape = dataclasses.replace(synth.LLAMA8B_STAGE, hidden=H)
    n_in = min(K, 64)  # distinct resident inputs, cycled
    hid = torch.from_numpy(np.stack([synth.hidden_in(shape, SEED, t, M) for t in range(n_in)]).view(np.int16)).to(dev)
    tok = torch.empty((K, M), dtype=torch.int32, device=dev)
    pm = torch.empty((K, M), dtype=torch.float32, device=dev)
    for t in range(W):
        pkg.head_top1(head, hid[t % n_in].data_ptr(), M, tok[0].data_ptr(), pm[0].data_ptr(), sptr)
    torch.cuda.synchronize()
    gpu_id = ""
    try:
        gpu_id = str(torch.cuda.get_device_properties(dev).uuid)
        if gpu_id and not gpu_id.startswith("GPU-"):
            gpu_id = "GPU-" + gpu_id
    except Exception:
        gpu_id = ""
    sampler = ClockSampler(gpu_id)
    time.sleep(0.3)
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    w0 = time.time()
    e0.record(stream)
    for t in range(K):
        pkg.head_top1(head, hid[t % n_in].data_ptr(), M, tok[t].data_ptr(), pm[t].data_ptr(), sptr)
    e1.record(stream)
    torch.cuda.synchronize()
    w1 = time.time()
    if dist:
        dist.barrier()
    ms = e0.elapsed_time(e1)
    sampler.stop()
    clocks = sampler.summary(w0, w1)
    ms = max_over_ranks(ms, dist, dev)
    # end to end: host hidden rows in, host (token, p_max) out, every call
    hosts = [synth.hidden_in(shape, SEED, 5000 + t, M) for t in range(min(K, 64))]
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for t in range(K):
        pkg.head_top1_host(head, hosts[t % len(hosts)], sptr)
    e2e_s = time.perf_counter() - t0
    e2e_s = max_over_ranks(e2e_s, dist, dev)
    pkg.head_destroy(head)
    if rank != 0:
        if dist:
            dist.destroy_process_group()
        return
    peaks = measured_peaks()
    peak = peaks.get("hbm_gbs")
    peak_note = "of measured" if peak else "of fallback"
    if not peak:
        peak = 6800.0
    call_bytes = hw.packed_bytes() + H * 2 + M * H * 2 + M * 8  # weights, norm, hidden rows, (token, p_max)
    call_s = ms / K / 1e3
    result = {
        "metric": HEAD_METRIC,
        "value": replica_throughput(world, K * M, ms / 1e3),
        "unit": "rows/s",
        "n_gpus": world,
        "steps": K,
        "warmup": W,
        "ms_per_step": ms / K,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "w4a16 (uint4 weights, fp16 activations, fp32 accumulate)",
        "data": "synthetic (seeded Gaussian lm_head quantised to uint4, fp16 N(0,1) hidden rows)",
        "config": {"workload": c["workload"], "rows_per_call": M,
                   "l2": "no flush: each call streams %.0f MB of packed weights, larger than the 129 MB L2" % (
                       hw.packed_bytes() / 1e6),
                   "parallelism": "replicas" if world > 1 else "single GPU", "seed": SEED},
        "call_alg_bytes": call_bytes,
        "roofline": {
            "kernel": "head_top1 call (norm + W4A16 projection + top-1 reduction; the projection dominates)",
            "bound": "hbm",
            "achieved": call_bytes / call_s / 1e9,
            "peak": peak,
            "unit": "GB/s",
            "frac": call_bytes / call_s / 1e9 / peak,
            "peak_note": "%s: MEASURED_PEAKS.json hbm_gbs; achieved = algorithmic bytes per call / CUDA-event "
                         "time per call" % peak_note,
            "traffic": profiled_traffic("head", args.config) if M == 1 else None,
            "traffic_note": "DRAM bytes of the projection kernel per call (ncu), M = 1",
        },
        "e2e": {"value": replica_throughput(world, K * M, e2e_s), "unit": "rows/s", "h2d_bytes_per_step": M * H * 2,
                "d2h_bytes_per_step": M * 8},
        "gpu_launches": 3 * K,
        "clocks": clocks,
    }
    if world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = head_cpu_baseline(hw, M, budget_s=args.cpu_budget)
    print(json.dumps(result), flush=True)
    if dist:
        dist.destroy_process_group()


def run_prefill(args, rank: int, world: int):
    """Prefill throughput (shard_prefill) and the tensor-core projection
    against the decode path's GEMV at small token counts."""
    import torch

    import paper_2608_19147_gb300 as pkg

    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", "0")))
    torch.cuda.set_device(dev)
    dist = None
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl", device_id=dev)
    c = CONFIGS[args.config]
    shape = c["shape"]
    if args.layers:
        shape = dataclasses.replace(shape, n_layers=args.layers)
    S = c["prefill_tokens"]
    K, W = args.steps, max(3, args.warmup)
    t0 = time.time()
    weights = synth.make_weights(shape, SEED)
    log("weights generated in %.1fs" % (time.time() - t0))
    sh = pkg.shard_create(pkg.make_config(shape), weights.layers, weights.embedding)
    stream = torch.cuda.current_stream(dev)
    sptr = stream.cuda_stream
    n_st = min(K + W, 16)  # states cycled (each call prefills an empty row; reset outside the timed region)
    sts = [pkg.kv_state_alloc(sh, 1, S + 8) for _ in range(n_st)]
    tok = torch.from_numpy(synth.token_ids(shape, SEED, 0, S).astype(np.int32)).to(dev)
    pos = torch.arange(S, dtype=torch.int32, device=dev)
    mask = torch.ones(S, dtype=torch.uint8, device=dev)
    out = torch.empty((S, shape.hidden), dtype=torch.int16, device=dev)

    def call(st):
        pkg.shard_prefill(sh, st, 0, None, tok.data_ptr(), S, pos.data_ptr(), mask.data_ptr(), S, out.data_ptr(), sptr)

    for i in range(W):
        call(sts[i % n_st])
    torch.cuda.synchronize()
    for st in sts:
        pkg.kv_state_reset(st, -1)
    gpu_id = ""
    try:
        gpu_id = str(torch.cuda.get_device_properties(dev).uuid)
        if gpu_id and not gpu_id.startswith("GPU-"):
            gpu_id = "GPU-" + gpu_id
    except Exception:
        gpu_id = ""
    ms_total, done = 0.0, 0
    clocks = None
    while done < K:
        n = min(n_st, K - done)
        sampler = ClockSampler(gpu_id)
        time.sleep(0.2)
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        w0 = time.time()
        e0.record(stream)
        for i in range(n):
            call(sts[i])
        e1.record(stream)
        torch.cuda.synchronize()
        w1 = time.time()
        sampler.stop()
        clocks = clocks or sampler.summary(w0, w1)
        ms_total += e0.elapsed_time(e1)
        done += n
        for st in sts[:n]:
            pkg.kv_state_reset(st, -1)
    pkg.shard_sync_status(sh, sptr)
    ms = max_over_ranks(ms_total, dist, dev)
    # the dominant kernel, the tensor-core projection, timed alone per 256-token chunk on layer 0
    chunk = 256
    proj = {}
    flops_chunk, ms_chunk = 0.0, 0.0
    for k, name in ((pkg.OP_QKV, "qkv"), (pkg.OP_O, "o"), (pkg.OP_GU, "gate_up"), (pkg.OP_DOWN, "down")):
        rows, Kin, _ = pkg.shard_debug_op_info(sh, 0, k)
        ld = (Kin + 127) // 128 * 128
        x = torch.zeros((chunk, ld), dtype=torch.int16, device=dev)
        x[:, :Kin] = torch.from_numpy(synth.hidden_in(dataclasses.replace(shape, hidden=Kin), SEED, 9, chunk).view(np.int16))
        y = torch.empty((chunk, rows), dtype=torch.float32, device=dev)
        for _ in range(3):
            pkg.shard_debug_gemm(sh, 0, k, x.data_ptr(), ld, chunk, y.data_ptr(), rows, sptr)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        reps = 20
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(reps):
            pkg.shard_debug_gemm(sh, 0, k, x.data_ptr(), ld, chunk, y.data_ptr(), rows, sptr)
        e1.record(stream)
        torch.cuda.synchronize()
        t_ms = e0.elapsed_time(e1) / reps
        fl = 2.0 * rows * Kin * chunk
        proj[name] = {"us_per_call": t_ms * 1e3, "tflops": fl / (t_ms * 1e9)}
        flops_chunk += fl
        ms_chunk += t_ms
    # the same projection at decode-sized token counts: the decode step's
    # mma.sync GEMV against the tcgen05 GEMM (gate|up of layer 0)
    rows, Kin, nbytes = pkg.shard_debug_op_info(sh, 0, pkg.OP_GU)
    ld = (Kin + 127) // 128 * 128
    cmp_m = {}
    for M in (1, 5, 8, 16):
        x = torch.zeros((M, ld), dtype=torch.int16, device=dev)
        x[:, :Kin] = torch.from_numpy(synth.hidden_in(shape, SEED, 11, M).view(np.int16))
        y = torch.empty((M, rows), dtype=torch.float32, device=dev)
        xk = x[:, :Kin].contiguous()
        res = {}
        for nm, fn in (("mma_sync_gemv", lambda: pkg.shard_debug_gemv(sh, 0, pkg.OP_GU, xk.data_ptr(), M, y.data_ptr(),
                                                                        rows, sptr)),
                       ("tcgen05_gemm", lambda: pkg.shard_debug_gemm(sh, 0, pkg.OP_GU, x.data_ptr(), ld, M,
                                                                       y.data_ptr(), rows, sptr))):
            for _ in range(3):
                fn()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            torch.cuda.synchronize()
            e0.record(stream)
            for _ in range(20):
                fn()
            e1.record(stream)
            torch.cuda.synchronize()
            t_ms = e0.elapsed_time(e1) / 20
            res[nm] = {"us_per_call": t_ms * 1e3, "weight_gbs": nbytes / (t_ms * 1e6)}
        cmp_m["M=%d" % M] = res
    for st in sts:
        pkg.kv_state_free(st)
    # end to end: token ids from pinned host memory in, hidden states out, every call
    htok = torch.from_numpy(synth.token_ids(shape, SEED, 0, S).astype(np.int32)).pin_memory()
    hout = torch.empty((S, shape.hidden), dtype=torch.int16).pin_memory()
    st = pkg.kv_state_alloc(sh, 1, S + 8)
    n_e2e = min(K, 4)
    e2e_s = 0.0
    for i in range(n_e2e):
        torch.cuda.synchronize()
        a = time.perf_counter()
        tok.copy_(htok, non_blocking=True)
        call(st)
        hout.copy_(out, non_blocking=True)
        torch.cuda.synchronize()
        e2e_s += time.perf_counter() - a
        pkg.kv_state_reset(st, -1)
    pkg.kv_state_free(st)
    pkg.shard_destroy(sh)
    if rank != 0:
        if dist:
            dist.destroy_process_group()
        return
    peaks = measured_peaks()
    peak = peaks.get("bf16_tflops")
    peak_note = "of measured (MEASURED_PEAKS.json bf16_tflops, burst; fp16 has the same dense rate)"
    if not peak:
        peak, peak_note = 1900.0, "of fallback (1.9 PFLOP/s bf16 burst)"
    result = {
        "metric": PREFILL_METRIC,
        "value": replica_throughput(world, K * S, ms / 1e3),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": K,
        "warmup": W,
        "ms_per_step": ms / K,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "w4a16 (uint4 weights, fp16 activations, fp32 accumulate)",
        "data": "synthetic (seeded Gaussian weights quantised to uint4; seeded token ids)",
        "config": {"workload": c["workload"], "tokens_per_call": S,
                   "shard": "%s: %d layers" % (shape.name, shape.n_layers),
                   "l2": "no flush: each call streams the %.2f GB of packed weights twice (two chunks)" % (
                       shape.packed_bytes_per_layer() * shape.n_layers / 1e9),
                   "parallelism": "replicas" if world > 1 else "single GPU", "seed": SEED},
        "roofline": {
            "kernel": "gemm_tc (W4A16 projection, tcgen05.mma kind::f16 M=128, N=128 tokens, accumulator in TMEM), "
                      "one 256-token chunk of each projection of layer 0, timed alone",
            "bound": "tensor",
            "achieved": flops_chunk / (ms_chunk * 1e9),
            "peak": peak,
            "unit": "TFLOP/s",
            "frac": flops_chunk / (ms_chunk * 1e9) / peak,
            "peak_note": peak_note,
            "traffic": None,
            "per_projection": proj,
        },
        "projection_gate_up_small_m": cmp_m,
        "e2e": {"value": replica_throughput(world, n_e2e * S, e2e_s), "unit": "tokens/s", "h2d_bytes_per_step": S * 4,
                "d2h_bytes_per_step": S * shape.hidden * 2},
        "gpu_launches": K * (2 + shape.n_layers * 11 * 2 + 1),
        "clocks": clocks,
    }
    if world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = prefill_cpu_baseline(shape, weights, budget_s=args.cpu_budget)
    print(json.dumps(result), flush=True)
    if dist:
        dist.destroy_process_group()


def prefill_cpu_baseline(shape, weights, budget_s: float = 20.0):
    """The oracle's step with a prompt of tokens as the new tokens of one
    request, on the host cores: a bounded prompt length, scaled to tokens/s."""
    import oracle
    oracle.build()
    oracle.set_threads(os.cpu_count() or 1)
    shard = oracle.OracleShard(shape, weights)
    n = 8
    st = shard.state(1, n + 8)
    tok = synth.token_ids(shape, SEED, 0, n)
    t0 = time.perf_counter()
    st.step([n], np.arange(n, dtype=np.int32), np.ones(n, np.uint8), token_ids=tok)
    dt = time.perf_counter() - t0
    return {"value": n / dt, "unit": "tokens/s", "cores": os.cpu_count() or 1, "kind": "oracle",
            "sample": "one %d-token prompt through the %d-layer stage (fp64 oracle, OpenMP over output rows), "
                      "%.1f s" % (n, shape.n_layers, dt)}


def run_reference(args, rank: int, world: int):
    if rank != 0:
        return
    c = CONFIGS[args.config]
    if "head" in c:
        H, V, g = c["head"]
        hw = synth.make_head(H, V, g, SEED)
        cb = head_cpu_baseline(hw, c["rows"], budget_s=float(os.environ.get("REFERENCE_BUDGET_S", "60")))
        print(json.dumps({
            "metric": HEAD_METRIC, "value": cb["value"], "unit": "rows/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1000.0 * c["rows"] / cb["value"], "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded Gaussian lm_head quantised to uint4)",
            "config": {"workload": c["workload"], "rows_per_call": c["rows"]}, "impl": "reference",
            "cpu_baseline": cb,
            "e2e": {"value": cb["value"], "unit": "rows/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        }), flush=True)
        return
    shape = c["shape"]
    weights = synth.make_weights(shape, SEED)
    if "prefill_tokens" in c:
        cb = prefill_cpu_baseline(shape, weights)
        print(json.dumps({
            "metric": PREFILL_METRIC, "value": cb["value"], "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1000.0 * c["prefill_tokens"] / cb["value"], "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded Gaussian weights quantised to uint4; seeded token ids)",
            "config": {"workload": c["workload"], "tokens_per_call": c["prefill_tokens"]}, "impl": "reference",
            "cpu_baseline": cb,
            "e2e": {"value": cb["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        }), flush=True)
        return
    budget = float(os.environ.get("REFERENCE_BUDGET_S", "120"))
    cb = cpu_baseline(args.config, weights, budget_s=budget, max_steps=args.steps, one_thread=False)
    result = {
        "metric": METRIC, "value": cb["value"], "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1000.0 * CONFIGS[args.config]["rows"] * c["n"] / cb["value"],
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f64", "data": "synthetic (seeded Gaussian weights quantised to uint4)",
        "config": {"workload": c["workload"], "rows_per_step": c["rows"] * c["n"]},
        "impl": "reference",
        "cpu_baseline": cb,
        "e2e": {"value": cb["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(result), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2048)
    ap.add_argument("--warmup", type=int, default=16)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--config", default="8b-decode", choices=list(CONFIGS))
    ap.add_argument("--no-cpu-baseline", action="store_true",
                    help="the workload's own line only: no CPU oracle leg and no other workloads")
    ap.add_argument("--no-other-workloads", action="store_true",
                    help="8b-decode at 1 GPU: skip measuring the other step workloads after the main line")
    ap.add_argument("--cpu-budget", type=float, default=20.0)
    ap.add_argument("--layers", type=int, default=0,
                    help="run only the stage's first N layers (profiling captures); default: the whole stage")
    args = ap.parse_args()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank, world)
    elif "head" in CONFIGS[args.config]:
        run_head(args, rank, world)
    elif "prefill_tokens" in CONFIGS[args.config]:
        run_prefill(args, rank, world)
    else:
        run_gpu(args, rank, world)


if __name__ == "__main__":
    main()
