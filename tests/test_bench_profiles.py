"""bench.py's link between the committed ncu summaries and the kernel sources
(CPU only): a summary's DRAM bytes per launch are reported as the roofline's
`traffic` only while the kernel source the counters were taken on is
unchanged -- a comment edit keeps them, any code change drops them."""
import os

import bench


def test_fingerprint_ignores_comments_and_blank_lines(tmp_path):
    a, b, c = tmp_path / "a.cu", tmp_path / "b.cu", tmp_path / "c.cu"
    a.write_text("int f() {\n  return 1;  // one\n}\n")
    b.write_text("// a header\n\nint f() {\n  return 1;\n}\n\n")
    c.write_text("int f() {\n  return 2;\n}\n")
    fa, fb, fc = (bench.code_fingerprint(str(p)) for p in (a, b, c))
    assert fa == fb != fc
    assert len(fa) == 16 and int(fa, 16) >= 0


def test_traffic_only_for_an_unchanged_kernel(tmp_path, monkeypatch):
    src = tmp_path / "paper_1612_08608_gb300" / "csrc"
    src.mkdir(parents=True)
    prof = tmp_path / "profiles"
    prof.mkdir()
    kernel = src / "k.cu"
    kernel.write_text("__global__ void k() {}\n")
    fp = bench.code_fingerprint(str(kernel))
    (prof / "k.txt").write_text("metric   value\n"
                                "dram_bytes_per_launch: 12345\n"
                                f"kernel_code_sha256_16: {fp}\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setitem(bench.TRAFFIC, ("w", "k"), ("k.txt", "k.cu"))
    assert bench.traffic_per_launch("w", "k") == 12345.0
    kernel.write_text("__global__ void k() {}  // a comment only\n")
    assert bench.traffic_per_launch("w", "k") == 12345.0
    kernel.write_text("__global__ void k() { int x = 0; }\n")
    assert bench.traffic_per_launch("w", "k") is None
    assert bench.traffic_per_launch("w", "not_mapped") is None


def test_committed_summaries_match_the_committed_kernels():
    # every summary the bench reads carries its DRAM figure and the
    # fingerprint of the kernel source it was captured on, and that source
    # has not changed since
    for (workload, kernel), (summary, source) in bench.TRAFFIC.items():
        path = os.path.join(bench.ROOT, "profiles", summary)
        txt = open(path).read()
        assert "dram_bytes_per_launch:" in txt and "kernel_code_sha256_16:" in txt, summary
        assert os.path.exists(os.path.join(bench.ROOT, "paper_1612_08608_gb300", "csrc", source))
        traffic = bench.traffic_per_launch(workload, kernel)
        assert traffic is not None and traffic > 0, (summary, source)
