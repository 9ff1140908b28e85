"""The numbers behind the bench line's roofline, checked on the CPU.

* algorithmic bytes: every tensor a c3 step (and step + commit) touches, counted
  from the tensors the synthetic inputs actually have and from the library's own
  state size, against bench.algorithmic_bytes;
* the DRAM-traffic record: keyed by a hash of the kernel's sources that ignores
  comments and whitespace, and dropped (null) as soon as the code changes;
* the reference arm's JSON line (the oracle on the host cores) and its rank rule;
* the clocks record, parsed from nvidia-smi's CSV.
"""
import json
import os
import shutil
import subprocess
import sys
import time

import bench
from paper_2608_06628_gb300 import build as B
from paper_2608_06628_gb300 import hybrid as H
from paper_2608_06628_gb300 import workloads as wk


def test_algorithmic_bytes_count_every_tensor_once():
    B.build()
    wl = wk.C3
    Q, K, V = wk.block_qkv(wl, "contract", "cpu")
    W, alpha = wk.params(wl)
    cfg = H.make_cfg(wl.d, wl.F, wl.Hq, wl.Hkv, wl.B, wl.io_dtype)
    state = H.hybrid_state_bytes(cfg) * wl.n_req
    nbytes = lambda t: t.numel() * t.element_size()
    ptrs = wl.n_req * 8
    ab = bench.algorithmic_bytes(wl, Q.element_size())
    # the step reads Q, K, V, W, alpha, the pointers and every state once, and writes O
    assert ab["attn"] == 2 * nbytes(Q) + nbytes(K) + nbytes(V) + nbytes(W) + nbytes(alpha) + state + ptrs
    # step + commit: the states are read once and written once
    assert ab["fused"] == ab["attn"] + state
    # the block commit: K, V, W, the pointers, every state read and written
    assert ab["commit"] == nbytes(K) + nbytes(V) + nbytes(W) + 2 * state + ptrs
    # the figure the bench line divides by for c3
    assert ab["fused"] == 88_736_320 and ab["attn"] == 54_919_744


def _fake_root(tmp_path, sources):
    root = tmp_path / "root"
    for rel in sources:
        dst = root / rel
        dst.parent.mkdir(parents=True, exist_ok=True)
        shutil.copy(os.path.join(bench.ROOT, rel), dst)
    (root / "profiles").mkdir(parents=True, exist_ok=True)
    return root


def test_traffic_record_follows_the_code_not_the_comments(tmp_path, monkeypatch):
    with open(os.path.join(bench.ROOT, "profiles", "traffic.json")) as fh:
        rec = json.load(fh)["hybrid_block_attn_commit"]
    root = _fake_root(tmp_path, rec["sources"])
    monkeypatch.setattr(bench, "ROOT", str(root))
    fake = dict(rec, source_sha=bench.source_sha(rec["sources"]))
    (root / "profiles" / "traffic.json").write_text(json.dumps({"hybrid_block_attn_commit": fake}))
    assert bench.recorded_traffic("hybrid_block_attn_commit", rec["workload"]) == rec["bytes_per_launch"]
    # another workload has no record
    assert bench.recorded_traffic("hybrid_block_attn_commit", "some other workload") is None
    kernel = root / rec["sources"][0]
    code = kernel.read_text()
    # a comment-only edit keeps the capture
    kernel.write_text("// a note\n" + code.replace("\n", "\n   \n", 3) + "\n/* another\n note */\n")
    assert bench.recorded_traffic("hybrid_block_attn_commit", rec["workload"]) == rec["bytes_per_launch"]
    # a change of code drops it
    kernel.write_text(code + "\nstatic int changed_kernel = 1;\n")
    assert bench.recorded_traffic("hybrid_block_attn_commit", rec["workload"]) is None


def test_committed_traffic_records_are_consistent():
    """Each committed capture adds up (a capture of an older build of a kernel is
    allowed: the bench line then reports its traffic as null)."""
    with open(os.path.join(bench.ROOT, "profiles", "traffic.json")) as fh:
        recs = json.load(fh)
    for name, rec in recs.items():
        assert all(os.path.exists(os.path.join(bench.ROOT, p)) for p in rec["sources"]), name
        assert rec["bytes_per_launch"] == rec["dram_read"] + rec["dram_write"], name
        ratio = rec["bytes_per_launch"] / rec["algorithmic_bytes"]
        assert abs(ratio - rec["traffic_over_algorithmic"]) < 1e-3, name


def _run_bench(args, env_extra=None):
    env = dict(os.environ, **(env_extra or {}))
    env.pop("CUDA_VISIBLE_DEVICES", None)
    return subprocess.run([sys.executable, "bench.py", *args], cwd=bench.ROOT, env=env,
                          capture_output=True, text=True, timeout=600)


def test_reference_arm_prints_one_contract_line():
    """bench.py --impl reference (the fp64 oracle on the host cores) prints one
    JSON line with the keys the driver reads, on the arm's own metric and config."""
    B.build()
    out = _run_bench(["--impl", "reference", "--config", "c1_fp32_tiny", "--steps", "2", "--warmup", "3"])
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [l for l in out.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, out.stdout
    line = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
                "cpu_baseline", "e2e"):
        assert key in line, key
    assert line["impl"] == "reference" and line["metric"] == bench.METRIC
    assert line["steps"] == 2 and line["warmup"] == 3 and line["n_gpus"] == 1
    assert line["higher_is_better"] is True and line["unit"] == "tokens/s" and line["value"] > 0
    assert line["config"]["workload"] == "c1_fp32_tiny"
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == line["value"] and cb["sample"]
    assert line["e2e"] == {"value": line["value"], "unit": "tokens/s",
                           "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_reference_arm_other_ranks_exit_without_work():
    out = _run_bench(["--impl", "reference", "--config", "c1_fp32_tiny", "--steps", "2", "--warmup", "3"],
                     {"RANK": "1", "LOCAL_RANK": "1", "WORLD_SIZE": "2"})
    assert out.returncode == 0, out.stderr[-2000:]
    assert out.stdout.strip() == ""


def test_warmup_below_three_is_refused():
    out = _run_bench(["--impl", "reference", "--config", "c1_fp32_tiny", "--steps", "1", "--warmup", "2"])
    assert out.returncode != 0 and "warmup" in out.stderr


def test_clock_sampler_reads_clocks_and_throttle_reasons(tmp_path, monkeypatch):
    """The clocks record of the bench line, from a stand-in nvidia-smi that prints
    the queried CSV fields: median SM clock, the maximum, and every throttle reason
    seen Active inside the window."""
    rows = ["0, 2070, 2070, 610.5, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active",
            "0, 1965, 2070, 1398.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active",
            "0, 2032, 2070, 1012.2, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active",
            "0, [N/A], 2070, [N/A], [N/A], [N/A], [N/A], [N/A], [N/A]",
            "0, 2070, 2070"]
    fake = tmp_path / "nvidia-smi"
    fake.write_text("#!/bin/sh\n" + "".join(f"echo '{r}'\n" for r in rows) + "exec sleep 30\n")
    fake.chmod(0o755)
    monkeypatch.setenv("PATH", f"{tmp_path}{os.pathsep}{os.environ['PATH']}")
    t0 = time.time()
    cs = bench.ClockSampler(None)
    cs.start()
    deadline = time.time() + 20
    while len(cs.samples) < 3 and time.time() < deadline:
        time.sleep(0.05)
    cs.stop()
    t1 = time.time()
    assert len(cs.samples) == 3   # the unparsable and short rows are skipped
    s = cs.summary(t0, t1)
    assert s["sm_mhz"] == 2032.0 and s["sm_max_mhz"] == 2070.0
    assert s["reasons"] == ["sw_power_cap"] and s["samples"] == 3
    # a window with no samples says so instead of reporting a clock
    far = cs.summary(t1 + 100, t1 + 101)
    assert far["sm_mhz"] is None and far["samples"] == 0


def test_algorithmic_bytes_of_the_context_configurations():
    """The per-call bytes the c2, c4 and c5 context lines divide by, from the
    shapes alone: Q and O once, K and V once, every state once per direction,
    W, alpha and the pointer array."""
    for wl, step, commit in ((wk.C2, None, None), (wk.C4, 84_934_976, 144_179_456),
                             (wk.C5, 1_351_616_576, 2_299_529_216)):
        n, Bk, Hq, Hkv, d, F = wl.n_req, wl.B, wl.Hq, wl.Hkv, wl.d, wl.F
        q, kv = n * Bk * Hq * d * 2, n * Bk * Hkv * d * 2
        state = n * Hkv * (2 * F * d + 2 * F) * 4
        w = Hkv * d * F * 2
        ab = bench.algorithmic_bytes(wl, 2)
        assert ab["attn"] == 2 * q + 2 * kv + state + w + 4 * Hq + 8 * n, wl.name
        assert ab["commit"] == 2 * kv + 2 * state + w + 8 * n, wl.name
        assert ab["fused"] == ab["attn"] + state, wl.name
        if step is not None:
            assert (ab["attn"], ab["commit"]) == (step, commit), wl.name
    assert bench.algorithmic_bytes(wk.C2, 2)["fused"] == 38_535_296
