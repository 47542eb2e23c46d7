"""The DRAM traffic that bench.py reports for the GEMM is the one its ncu
summary under profiles/ records (read + write bytes of one launch)."""

import importlib.util
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_gemm_traffic_matches_profile():
    spec = importlib.util.spec_from_file_location("bench", os.path.join(ROOT, "bench.py"))
    bench = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(bench)
    text = open(os.path.join(ROOT, "profiles", "gemm_ts_qkv_m4608_k4096_n12288.md")).read()
    m = re.search(r"traffic \(read \+ write\) per launch \| ([0-9.]+) MB", text)
    assert m, "the summary states the per-launch traffic"
    read = float(re.search(r"dram__bytes_read.sum` \| ([0-9.]+) MB", text).group(1))
    write = float(re.search(r"dram__bytes_write.sum` \| ([0-9.]+) MB", text).group(1))
    assert abs(read + write - float(m.group(1))) < 0.01
    assert abs(bench.GEMM_TRAFFIC_BYTES[("ts", "qkv_m4608_k4096_n12288")] / 1e6 - float(m.group(1))) < 0.01
