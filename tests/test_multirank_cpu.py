"""bench.py host logic on CPU.  The N>1 replica path: two gloo ranks (127.0.0.1), each with its
own step time; the reported time is the max over ranks and the throughput counts the
tokens of every replica.  The reference arm runs on rank 0 only."""
import importlib.util
import io
import os
import socket
import contextlib

import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench", os.path.join(ROOT, "bench.py"))
    b = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(b)
    return b


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        b = _bench()
        ms = 10.0 + 5.0 * rank  # rank 1 is the slow replica
        dist.barrier()
        m = b.max_over_ranks(ms)
        tok = b.whole_job_tokens_per_s(16384, world, m)
        # the reference arm prints only on rank 0
        args = type("A", (), {"cpu_tokens": 1, "ref_tokens": 1, "warmup": 0, "steps": 0,
                              "gpus": world})()
        buf = io.StringIO()
        if rank != 0:
            with contextlib.redirect_stdout(buf):
                b.run_reference(args, None)
        q.put((rank, m, tok, buf.getvalue()))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_max_time_and_sum_tokens():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, m, tok, out in res:
        assert m == 15.0
        assert abs(tok - 16384 * 2 / 0.015) < 1e-6
        assert out == ""


def test_single_rank_needs_no_process_group():
    b = _bench()
    assert b.max_over_ranks(12.5) == 12.5
    assert b.whole_job_tokens_per_s(100, 1, 10.0) == 10000.0


def test_reference_arm_prints_the_contract_line():
    """bench.py --impl reference (the oracle on the host cores) prints one JSON line with
    the keys of the bench contract, for the tiny workload in a couple of seconds."""
    import json
    import subprocess
    import sys
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--workload", "tiny", "--steps", "3", "--warmup", "3"],
                         capture_output=True, text=True, timeout=300, cwd=ROOT)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [l for l in out.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for k in ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
              "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
              "cpu_baseline", "e2e"):
        assert k in d, k
    assert d["impl"] == "reference" and d["steps"] == 3 and d["warmup"] == 3
    assert d["value"] > 0 and d["cpu_baseline"]["value"] == d["value"]
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["e2e"]["value"] == d["value"] and d["e2e"]["h2d_bytes_per_step"] == 0
    assert d["config"]["workload"] == "tiny-f32"
    # the oracle runs one token per host thread at a time: the sample keeps every thread
    # busy (four tokens per thread for a 6-step run, capped at the workload's 128 tokens)
    n = int(d["cpu_baseline"]["sample"].split(" of ")[0])
    assert n == min(128, 4 * d["cpu_baseline"]["cores"])


def test_reference_arm_loads_no_product_code():
    """The oracle arm loads the oracle's library and nothing of the CUDA path: its inputs
    come from synth.py, which sits outside the library package, and it never builds or
    imports the binding (so libfpo.so is not mapped into the process)."""
    import json
    import subprocess
    import sys
    code = (
        "import json, runpy, sys\n"
        "sys.argv = ['bench.py', '--impl', 'reference', '--workload', 'tiny', '--steps', '1',"
        " '--warmup', '3']\n"
        "runpy.run_path('bench.py', run_name='__main__')\n"
        "maps = open('/proc/self/maps').read().splitlines()\n"
        "libs = sorted({l.split()[-1].rsplit('/', 1)[-1] for l in maps"
        " if l.endswith('.so') and ('libfpo' in l or 'liboracle' in l)})\n"
        "print('LOADED ' + json.dumps({'libs': libs, 'binding':"
        " 'paper_2608_14563_gb300' in sys.modules}))\n")
    out = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, timeout=300,
                         cwd=ROOT)
    assert out.returncode == 0, out.stderr[-2000:]
    line = [l for l in out.stdout.splitlines() if l.startswith("LOADED ")][0]
    d = json.loads(line[len("LOADED "):])
    assert d == {"libs": ["liboracle.so"], "binding": False}, d
    ref = json.loads([l for l in out.stdout.splitlines() if l.startswith("{")][0])
    assert ref["ms_per_step_kind"] == "extrapolated" and "extrapolated" in ref["timing"]


def test_bench_rejects_fewer_than_three_warmups():
    import subprocess
    import sys
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--workload", "tiny", "--steps", "1", "--warmup", "2"],
                         capture_output=True, text=True, timeout=120, cwd=ROOT)
    assert out.returncode != 0 and "warmup" in out.stderr


def test_end_to_end_copy_schedule():
    """Per-phase copies while a step's copy fits beside the error signal's GEMMs (the
    OLMo shape: 14.4 ms of copy, 16.3 ms of GEMMs), else one launch per step (the Falcon
    shape: 51 ms of copy, 34 ms of GEMMs); an explicit choice is kept."""
    b = _bench()
    assert b.copy_schedule("auto", 14.4, 16.3) == "sm"
    assert b.copy_schedule("auto", 51.1, 33.4) == "sm1"
    assert b.copy_schedule("auto", 16.3, 16.3) == "sm"
    for m in ("sm", "sm1", "ce"):
        assert b.copy_schedule(m, 51.1, 33.4) == m


def test_committed_traffic_summary_matches_the_gemm_sources():
    """The bench's roofline.traffic comes from profiles/traffic.json only while its source
    digest matches the GEMM sources: a kernel change without a new capture reads null."""
    b = _bench()
    cfg = {"workload": "olmo2-7b-shaped", "algo": "direct", "gemm_variant": 2, "t_chunk": 8192,
           "window_stress": False}
    got = {k: b.load_traffic(k, cfg) for k in ("logits_lse_pass", "projection", "layer_update")}
    assert all(v is not None and v > 0 for v in got.values()), got
    assert b.load_traffic("logits_lse_pass", dict(cfg, t_chunk=4096)) is None
