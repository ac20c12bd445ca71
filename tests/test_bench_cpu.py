"""Host logic of bench.py's roofline traffic on CPU: DRAM bytes come from
ncu captures keyed by a hash of the kernel's sources, so an edited kernel
reports null traffic until it is captured again; the attention capture (8
pairs) scales with the benched pair count."""
import os
import shutil
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_every_traffic_entry_names_known_sources():
    for (config, kind, digest), value in bench.NCU_TRAFFIC.items():
        assert kind in bench.KERNEL_FILES, (config, kind)
        assert len(digest) == 16 and all(ch in "0123456789abcdef" for ch in digest)
        assert value > 0


def test_traffic_follows_the_source_hash(tmp_path, monkeypatch):
    csrc = os.path.join(ROOT, "paper_2608_30877_gb300", "csrc")
    fake = tmp_path / "paper_2608_30877_gb300" / "csrc"
    fake.mkdir(parents=True)
    for kind in bench.KERNEL_FILES.values():
        for name in kind:
            shutil.copy(os.path.join(csrc, name), fake / name)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    before = {k: bench.kernel_source_hash(k) for k in bench.KERNEL_FILES}
    assert before == {k: bench.kernel_source_hash(k) for k in bench.KERNEL_FILES}  # stable
    stack = bench.ncu_traffic("stack", 65536)
    # any edit of a kernel source changes its hash and drops the stale number
    with open(fake / "ts_gemm.cu", "a") as f:
        f.write("\n// edited\n")
    assert bench.kernel_source_hash("ts") != before["ts"]
    assert bench.ncu_traffic("stack", 65536) is None
    assert bench.kernel_source_hash("gemv") == before["gemv"]
    if stack is not None:
        assert stack == bench.NCU_TRAFFIC[("stack", "ts", before["ts"])]


def test_attention_traffic_scales_with_pairs():
    t8 = bench.ncu_traffic("attention", 0, 8)
    if t8 is None:  # sources changed since the capture
        return
    assert bench.ncu_traffic("attention", 0, 64) == t8 * 8
    assert bench.ncu_traffic("topk", 0) is None
    # M = 9..16 read the M = 16 capture, M = 17..32 the tensor-core kernel's
    h = bench.kernel_source_hash("gemv")
    assert bench.ncu_traffic("gemv", 12) == bench.NCU_TRAFFIC.get(("gemv16", "gemv", h))
    assert bench.ncu_traffic("gemv", 3) == bench.NCU_TRAFFIC.get(("gemv", "gemv", h))
    t = bench.kernel_source_hash("ts")
    for c in ("mlp_up", "mlp_down", "qkv"):
        assert bench.ncu_traffic(c, 8192) == bench.NCU_TRAFFIC.get((c, "ts", t))
    assert bench.ncu_traffic("mlp_swiglu", 8192) is None
