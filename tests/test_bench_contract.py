"""The numbers behind the bench line's roofline, checked on the CPU.

* algorithmic bytes: every tensor a c3 step (and step + commit) touches, counted
  from the tensors the synthetic inputs actually have and from the library's own
  state size, against bench.algorithmic_bytes;
* the DRAM-traffic record: keyed by a hash of the kernel's sources that ignores
  comments and whitespace, and dropped (null) as soon as the code changes.
"""
import json
import os
import shutil

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
