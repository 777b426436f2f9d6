"""bench.py's default line also carries the other step workloads, each
measured by `bench.py --config <name>` in a child process after the main
line's timed region.  Host logic only (no GPU): which runs take them, how a
child's line is read, that a failing child leaves an error entry instead of
breaking the main line, and that the children never see the launcher's rank
variables (each is a single-GPU run of its own)."""
import argparse
import json
import sys

import pytest

import bench


def _args(**kw):
    base = dict(config="8b-decode", layers=0, no_cpu_baseline=False, no_other_workloads=False)
    base.update(kw)
    return argparse.Namespace(**base)


def test_which_runs_measure_the_other_workloads():
    assert bench.want_other_workloads(_args(), 1)
    assert not bench.want_other_workloads(_args(), 2)                      # replicas under torchrun
    assert not bench.want_other_workloads(_args(config="70b-decode"), 1)   # a child itself
    assert not bench.want_other_workloads(_args(no_cpu_baseline=True), 1)  # the bare line (profiling)
    assert not bench.want_other_workloads(_args(no_other_workloads=True), 1)
    assert not bench.want_other_workloads(_args(layers=4), 1)
    # every other step workload, and only step workloads
    names = [c for c, _ in bench.OTHER_WORKLOADS]
    assert sorted(names) == ["70b-decode", "70b-verify", "8b-microbatch", "8b-verify"]
    assert all("shape" in bench.CONFIGS[c] and "head" not in bench.CONFIGS[c] for c in names)


def test_child_lines_are_read_and_failures_recorded(monkeypatch):
    line = {"config": {"workload": "w"}, "value": 12.5, "unit": "tokens/s", "ms_per_step": 2.0, "steps": 64,
            "roofline": {"achieved": 3000.0, "frac": 0.44, "peak": 6796.5}, "e2e": {"value": 12.0},
            "clocks": {"sm_mhz": 2070.0}, "gpu_launches": 64}

    def fake(cfg, steps):
        if cfg == "8b-verify":
            return [sys.executable, "-c", "import sys; print('boom', file=sys.stderr); sys.exit(3)"]
        return [sys.executable, "-c", "print('log line'); print(%r)" % json.dumps(line)]

    monkeypatch.setattr(bench, "_child_cmd", fake)
    out = bench.other_workloads(timeout_s=60)
    assert set(out) == {c for c, _ in bench.OTHER_WORKLOADS}
    assert out["8b-verify"] == {"error": "exit 3: boom"}
    ok = out["70b-decode"]
    assert ok["value"] == 12.5 and ok["frac"] == 0.44 and ok["e2e"] == 12.0 and ok["gpu_launches"] == 64
    json.dumps(out)  # rides in the JSON line


def test_a_child_that_hangs_is_cut_off(monkeypatch):
    monkeypatch.setattr(bench, "OTHER_WORKLOADS", (("70b-decode", 64),))
    monkeypatch.setattr(bench, "_child_cmd", lambda c, s: [sys.executable, "-c", "import time; time.sleep(30)"])
    out = bench.other_workloads(timeout_s=1)
    assert out["70b-decode"]["error"].startswith("TimeoutExpired")


def test_children_do_not_inherit_launcher_ranks(monkeypatch):
    for k, v in (("RANK", "0"), ("WORLD_SIZE", "1"), ("LOCAL_RANK", "0"), ("MASTER_PORT", "29500"),
                 ("TORCHELASTIC_RUN_ID", "x"), ("KEEP_ME", "1")):
        monkeypatch.setenv(k, v)
    env = bench._child_env()
    assert "KEEP_ME" in env
    assert not any(k in env for k in ("RANK", "WORLD_SIZE", "LOCAL_RANK", "MASTER_PORT", "TORCHELASTIC_RUN_ID"))
    cmd = bench._child_cmd("8b-verify", 128)
    assert cmd[-7:] == ["--config", "8b-verify", "--steps", "128", "--warmup", "3", "--no-cpu-baseline"]


def test_children_share_one_overall_deadline(monkeypatch):
    monkeypatch.setattr(bench, "_child_cmd", lambda c, s: [sys.executable, "-c", "import time; time.sleep(30)"])
    out = bench.other_workloads(timeout_s=2, total_s=13)
    errs = [out[c]["error"] for c, _ in bench.OTHER_WORKLOADS]
    assert errs[0].startswith("TimeoutExpired") and any(e.startswith("skipped") for e in errs)
