"""Host-side logic of bench.py: the kernel-source hash behind the recorded ncu traffic, the
traffic lookup, and the names of the kernels each layer workload launches."""
import json
import os

import bench
from paper_2412_06355_gb300 import workloads


def test_comment_only_edits_keep_the_source_hash():
    src = "int f(int a) {\n  return a + 1;  // add one\n}\n/* block\n comment */\n\n"
    same = "int f(int a) {\n  return a + 1;\n}\n"
    changed = "int f(int a) {\n  return a + 2;\n}\n"
    assert bench._strip_comments(src) == bench._strip_comments(same)
    assert bench._strip_comments(src) != bench._strip_comments(changed)


def test_recorded_traffic_needs_the_current_source_hash(tmp_path, monkeypatch):
    h = bench.kernel_source_hash()
    rec = {"conv": {"k": {"dram_bytes_per_launch": 123.0, "source_hash": h}},
           "old": {"k": {"dram_bytes_per_launch": 456.0, "source_hash": "0" * 16}}}
    os.makedirs(tmp_path / "profiles")
    (tmp_path / "profiles" / "traffic.json").write_text(json.dumps(rec))
    # the hash is taken over the library sources under ROOT: point ROOT at a copy of them
    os.symlink(os.path.join(bench.ROOT, "paper_2412_06355_gb300"), tmp_path / "paper_2412_06355_gb300")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.kernel_source_hash() == h
    assert bench.recorded_traffic("k", "conv") == 123.0
    assert bench.recorded_traffic("k", "old") is None          # kernels changed since the capture
    assert bench.recorded_traffic("other", "conv") is None


def test_committed_traffic_record_names_kernels_the_layers_launch():
    with open(os.path.join(bench.ROOT, "profiles", "traffic.json")) as f:
        rec = json.load(f)
    for wl, kernels in rec.items():
        assert set(kernels) <= set(bench.kernel_names(workloads.WORKLOADS[wl])), wl


def test_kernel_names_follow_the_library_plan():
    W = workloads.WORKLOADS
    assert bench.kernel_names(W["conv"]) == ("dendsn_forward_kernel", "dendsn_backward_kernel")
    # 4-step rows of 8 float32 compartments on two lanes: two rows per thread
    assert bench.kernel_names(W["token_dbg"]) == ("dendsn_forward_kernel", "dendsn_backward_rowpair_kernel")
    assert bench.kernel_names(W["token_dbg"].with_(T=5))[1] == "dendsn_backward_kernel"
    assert bench.kernel_names(W["event"]) == ("dendsn_forward_kernel", "dendsn_backward_kernel")
    # rows of one full 8-step chunk, 8 bf16 compartments on one lane
    assert bench.kernel_names(W["deepconv_bf16"])[1] == "dendsn_backward_phased_vs_kernel"
    assert bench.kernel_names(W["deepconv_bf16"].with_(dtype="f32"))[1] == "dendsn_backward_phased_kernel"
    # ... but not with the residual term, nor in the paper layout
    assert bench.kernel_names(W["deepconv_bf16"].with_(residual=True))[1] == "dendsn_backward_kernel"
    assert bench.kernel_names(W["deepconv_bf16"].with_(layout="paper"))[1] == "dendsn_backward_kernel"
    # the paper layout with 32-aligned positions stages the forward per warp
    assert bench.kernel_names(W["conv_paper_p4b2"])[0] == "dendsn_forward_staged_kernel"
    # long horizons on a handful of neurons: the time-parallel kernels
    assert bench.kernel_names(W["l5pc"]) == ("tp_forward_kernel", "tp_backward_kernel")
    assert bench.kernel_names(W["long_t"])[1] == "dendsn_backward_kernel"
