"""The bench's CPU-side paths: the reference arm (the oracle timed on the host)
end to end on a small workload, and the roofline helpers.  No GPU."""
import argparse
import io
import json
import os
import sys
from contextlib import redirect_stdout

ROOT = os.path.abspath(os.path.join(os.path.dirname(__file__), ".."))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2609_13804_gb300 import synth as S  # noqa: E402


def test_reference_arm_prints_one_complete_line():
    w = S.tiny_workload(71, [24, 16], [4, 3], D=32, D_text=64, d=64, n_heads=4, n_kv_heads=2, head_dim=16, ffn=96,
                        n_layers=2)
    buf = io.StringIO()
    with redirect_stdout(buf):
        bench.run_reference(argparse.Namespace(steps=2, warmup=1, gpus=1), w=w)
    lines = [l for l in buf.getvalue().splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["higher_is_better"] is False
    assert d["samples_timed"] == 2 and d["value"] > 0 and d["value"] == d["ms_per_step"]
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["extrapolated"] is True and d["e2e"]["h2d_bytes_per_step"] == 0
    assert d["config"]["images"] == 2 and d["config"]["layers"] == 2


def test_attention_roofline_entry():
    pk = {"bf16": 2000.0, "source": "measured"}
    r = bench.attention_roofline(2.0, 2.0e12, 32, pk, None)
    assert r["bound"] == "tensor" and abs(r["achieved"] - 1000.0) < 1e-9 and abs(r["frac"] - 0.5) < 1e-12
    assert "long" not in r
    wl = {"internvl3-tiles-b4": {"full_prefix": {"attention_tflops": 800.0, "attention_frac_of_bf16_burst": 0.4}}}
    r = bench.attention_roofline(2.0, 2.0e12, 32, pk, wl)
    assert r["long"]["frac"] == 0.4


def test_traffic_figures_follow_the_kernel_sources():
    # the committed ncu traffic figures belong to the current sources, or are withheld
    g, a = bench.gemm_traffic(), bench.attn_traffic()
    assert g in (None, bench.GEMM_TRAFFIC["bytes_per_launch"])
    assert a in (None, bench.ATTN_TRAFFIC["bytes_per_launch"])
