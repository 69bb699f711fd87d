"""Host-side rules of bench.py that need no GPU: where the bench line's
`roofline.traffic` comes from, and that the committed ncu summaries carry
what that rule reads."""
import glob
import os
import re
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _summary(digest: str, nbytes: int) -> str:
    return (f"# a summary\n\nkernel_source_sha256: {digest}\n"
            f"dram_bytes_per_launch: {nbytes}\n")


def test_traffic_is_read_only_while_the_kernel_source_is_unchanged(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "PROFILE_DIR", str(tmp_path))
    path = tmp_path / "stream_topk_qwen3-0.6b_b1_k50.md"
    # no summary: no traffic, no profile
    assert bench.profiled_traffic("stream_topk", "qwen3-0.6b", 1, 50) == (None, None)
    # a summary of the current sources: its bytes
    path.write_text(_summary(bench.kernel_source_digest("stream_topk"), 311276032))
    assert bench.profiled_traffic("stream_topk", "qwen3-0.6b", 1, 50) == (311276032, str(path))
    # a summary of other sources: null traffic, the summary still named
    path.write_text(_summary("0" * 16, 311276032))
    assert bench.profiled_traffic("stream_topk", "qwen3-0.6b", 1, 50) == (None, str(path))
    # a summary without the two fields: null traffic
    path.write_text("# a summary\n")
    assert bench.profiled_traffic("stream_topk", "qwen3-0.6b", 1, 50) == (None, str(path))
    # another batch or k is another launch shape: not this summary
    path.write_text(_summary(bench.kernel_source_digest("stream_topk"), 311276032))
    assert bench.profiled_traffic("stream_topk", "qwen3-0.6b", 4, 50) == (None, None)
    assert bench.profiled_traffic("stream_topk", "qwen3-0.6b", 1, 1) == (None, None)


def test_digests_cover_each_kernels_sources():
    for kernel, files in bench.KERNEL_SOURCES.items():
        for f in files:
            assert os.path.exists(os.path.join(ROOT, "paper_2608_27460_gb300", "csrc", f)), (kernel, f)
        assert re.fullmatch(r"[0-9a-f]{16}", bench.kernel_source_digest(kernel))
    # the streaming and tensor-core kernels are built from different sources
    assert bench.kernel_source_digest("stream_topk") != bench.kernel_source_digest("tc_topk")


def test_committed_summaries_are_readable():
    """Every ncu summary names a kernel bench.py knows, a workload, batch
    and k in its file name, the digest and bytes bench.py reads, and the
    commands that made it, which run committed files only."""
    files = sorted(glob.glob(os.path.join(ROOT, "profiles", "*.md")))
    assert files
    for f in files:
        name = os.path.basename(f)
        m = re.fullmatch(r"(stream_topk_e4m3|tc_topk_e4m3|stream_topk|tc_topk)_(.+)_b(\d+)_k(\d+)\.md", name)
        assert m, name
        assert m.group(2) in bench.synth.HEADS, name
        text = open(f).read()
        assert re.search(r"kernel_source_sha256:\s*[0-9a-f]{16}", text), name
        nbytes = int(re.search(r"dram_bytes_per_launch:\s*([0-9]+)", text).group(1))
        shape = bench.synth.HEADS[m.group(2)]
        w = shape.V * shape.d * (1 if "e4m3" in m.group(1) else 2)
        assert w <= nbytes <= 1.1 * w + 64e6, (name, nbytes, w)  # W once, plus small extras
        assert "ncu " in text and "--clock-control none" in text, name
        for cmd in re.findall(r"python (\S+\.py)", text):
            assert os.path.exists(os.path.join(ROOT, cmd)), (name, cmd)
