"""The multi-GPU path's host logic with two gloo ranks on the CPU.

Multi-GPU runs are independent replicas (weak scaling): every rank runs the whole sweep on
its own seeded problem and nothing crosses ranks on the data path.  What crosses is the
timing: the slowest rank's time sets the job's, and the job's throughput counts every rank's
meta-steps.  The CPU reference arm runs on rank 0 alone."""
import io
import json
import os
import socket
import sys
from contextlib import redirect_stdout

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, ws, port, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(ws), LOCAL_RANK=str(rank))
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    try:
        import bench
        from paper_2505_00793_gb300 import synth
        assert bench._dist() == (ws, rank, rank)
        # rank r took (10 + 5 r) ms in total over 4 steps
        ms, value = bench._job_rate(10.0 + 5.0 * rank, 4, ws, "cpu")
        mx = bench._max_over_ranks(float(rank), ws, "cpu")
        w = bench._replica_workload(synth.WORKLOADS["tiny"], rank)
        theta0 = synth.make_inputs(w).theta0
        # the reference arm: ranks other than 0 return at once and print nothing
        out = io.StringIO()
        rc = None
        if rank != 0:
            with redirect_stdout(out):
                rc = bench.run_reference(type("A", (), {"warmup": 1, "steps": 1, "gpus": ws})())
        q.put((rank, ms, value, mx, w.seed, float(theta0[0]), rc, out.getvalue()))
    finally:
        dist.destroy_process_group()


def test_two_rank_replicas():
    torch = pytest.importorskip("torch")
    mp = torch.multiprocessing.get_context("spawn")
    q = mp.Queue()
    port = _free_port()
    procs = [mp.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=240) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, ms0, v0, mx0, s0, t0, _, _), (r1, ms1, v1, mx1, s1, t1, rc1, out1) = res
    # the slowest rank's 15 ms over 4 steps, and both ranks' steps in the throughput
    assert ms0 == ms1 == pytest.approx(15.0 / 4)
    assert v0 == v1 == pytest.approx(2 * 1000.0 / (15.0 / 4))
    assert mx0 == mx1 == 1.0
    # each replica draws its own problem
    assert s1 == s0 + 1 and t0 != t1
    assert rc1 == 0 and out1 == ""


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench._job_rate(12.0, 3, 1, "cpu") == (4.0, 250.0)
    assert bench._max_over_ranks(7.5, 1, "cpu") == 7.5
    from paper_2505_00793_gb300 import synth
    w = synth.WORKLOADS["tiny"]
    assert bench._replica_workload(w, 0) is w


def _ref_args(**kw):
    a = {"warmup": 0, "steps": 1, "gpus": 1}
    a.update(kw)
    return type("A", (), a)()


def _tiny_large_decoder():
    """A tiny decoder under the name of the sampled workload (same code path, seconds)."""
    from paper_2505_00793_gb300 import synth
    return synth.decoder("decoder_large", 16, 2, 32, 2, 32, 8, B=2, T=3, B_outer=2,
                         momentum=0.9, meta_kind=synth.EXAMPLE_WEIGHTS | synth.SCALAR_LOGLR)


@pytest.mark.parametrize("sampled", [True, False])
def test_reference_line_contract(monkeypatch, sampled):
    """``--impl reference`` prints one JSON line with the contract's keys (the oracle timed on
    a tiny stand-in workload here, to keep the CPU suite short); its per-step time times the
    step count is the timed wall time."""
    sys.path.insert(0, ROOT)
    import bench
    from paper_2505_00793_gb300 import synth
    w = _tiny_large_decoder() if sampled else synth.WORKLOADS["tiny"].with_(T=16)
    monkeypatch.setitem(synth.WORKLOADS, bench.WORKLOAD, w)
    out = io.StringIO()
    with redirect_stdout(out):
        rc = bench.run_reference(_ref_args(workload=bench.WORKLOAD, steps=4, warmup=1))
    assert rc == 0
    d = json.loads(out.getvalue().strip().splitlines()[-1])
    assert d["impl"] == "reference" and d["unit"] == "meta-steps/s" and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["value"] == d["value"]
    assert d["higher_is_better"] is True and d["steps"] == 4
    if sampled:
        assert d["ms_per_step"] * 4 / 1000.0 <= d["timed_wall_s"] * 1.05 + 0.05


def test_cpu_baseline_whole_oracle_repeats_to_its_minimum_time():
    sys.path.insert(0, ROOT)
    import bench
    from paper_2505_00793_gb300 import synth
    c = bench.cpu_baseline(synth.WORKLOADS["tiny"], min_seconds=0.2)
    assert c["kind"] == "oracle" and c["value"] > 0 and c["cores"] >= 1
    assert "whole oracle meta-gradients" in c["sample"]


def test_cpu_baseline_units_scale_to_a_meta_step(monkeypatch):
    """The sampled baseline: one unit of each kind, meta-step time B T (rollout + reverse)
    + B_outer outer."""
    sys.path.insert(0, ROOT)
    import bench
    w = _tiny_large_decoder()
    calls = []

    def fake_unit(w_, kind):
        calls.append(kind)
        return {"rollout": 0.5, "reverse": 1.5, "outer": 0.25}[kind]

    monkeypatch.setattr(bench, "oracle_unit", fake_unit)
    c = bench.cpu_baseline(w)
    assert sorted(calls) == sorted(bench.UNIT_KINDS)
    assert c["value"] == pytest.approx(1.0 / (w.B * w.T * 2.0 + w.B_outer * 0.25))
    # the real units run on one sequence of one step
    monkeypatch.undo()
    for k in bench.UNIT_KINDS:
        assert bench.oracle_unit(w, k) > 0
