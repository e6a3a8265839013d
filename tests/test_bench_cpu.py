"""bench.py's host-side bookkeeping, without a GPU: the ncu traffic figure of the roofline entry
is reported only while the sources it was captured from are unchanged, and the hash that decides
it covers every source the kernel is built and planned from."""
import os
import shutil

import bench


def test_traffic_is_reported_only_for_the_captured_sources(monkeypatch):
    h = bench.source_hash("attention")
    monkeypatch.setitem(bench.NCU_TRAFFIC, ("attention", 99), (123_456, h))
    assert bench.ncu_traffic("attention", 99) == 123_456
    monkeypatch.setitem(bench.NCU_TRAFFIC, ("attention", 99), (123_456, "0" * 16))
    assert bench.ncu_traffic("attention", 99) is None       # captured from other sources
    assert bench.ncu_traffic("attention", 98) is None       # never captured


def test_source_hash_follows_every_listed_source(monkeypatch, tmp_path):
    src = os.path.join(bench.ROOT, "paper_2502_16002_gb300", "csrc")
    dst = tmp_path / "paper_2502_16002_gb300" / "csrc"
    shutil.copytree(src, dst)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    for kernel, files in bench.KERNEL_SOURCES.items():
        base = bench.source_hash(kernel)
        for f in files:
            p = dst / f
            text = p.read_bytes()
            p.write_bytes(text + b"\n// changed\n")
            assert bench.source_hash(kernel) != base, (kernel, f)
            p.write_bytes(text)
        assert bench.source_hash(kernel) == base
    # the zero-copy kernels are instantiations of the same sources
    assert bench.KERNEL_SOURCES["attention_pool_values"] == bench.KERNEL_SOURCES["attention"]
    assert bench.KERNEL_SOURCES["reencode_keys"] == bench.KERNEL_SOURCES["reencode"]


def test_whole_job_rate_counts_every_rank():
    # 3.5 ms per step, 8 queries per rank, 4 ranks: 32 queries in 3.5 ms
    assert abs(bench.whole_job_us_per_query(3.5, 8, 4) - 3500.0 / 32) < 1e-9
