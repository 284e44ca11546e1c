"""The benchmark's host side on the CPU: the reference arm (the oracle on the
host cores) prints one JSON line with every key of the benchmark contract, and
the algorithmic byte counts the roofline divides by are the large stream's
(1.372 GB for each forward call, 1.087 GB for each backward call, 268 MB for
the projection of W_o [8192, 8192])."""
import importlib.util
import json
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)

KEYS = ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
        "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
        "cpu_baseline", "e2e")


def _bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_reference_arm_prints_one_contract_line():
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    out = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--steps", "1",
                          "--warmup", "0", "--cpu-seconds", "1"], cwd=ROOT, env=env,
                         capture_output=True, text=True, timeout=900)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [ln for ln in out.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    line = json.loads(lines[0])
    for key in KEYS:
        assert key in line, key
    assert line["impl"] == "reference"
    assert line["unit"] == "tokens/s" and line["higher_is_better"] is True
    assert line["value"] > 0 and line["ms_per_step"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["d2h_bytes_per_step"] == 0
    assert line["config"]["T"] == 65536 and line["config"]["d"] == 8192


def test_algorithmic_bytes_of_the_large_stream():
    ab = _bench().algorithmic_bytes(T=65536, d=8192, k=82, n=4096, u=13284, m_cols=8192)
    assert ab["sn_compress_fwd"] == ab["sn_decompress_fwd"] == 1371930624
    assert ab["sn_compress_bwd"] == ab["sn_decompress_bwd"] == 1087176704
    assert ab["sn_project_weight"] == 268435456


def test_paper_context_of_the_large_stream():
    ctx = _bench().paper_context(T=65536, d=8192, k=82, codec_ms=1.0)
    assert ctx["wire_bytes_per_step"] == 2 * 65536 * 82 * 2
    assert abs(ctx["compression_ratio"] - 8192 / 82) < 1e-9
    assert abs(ctx["compression_pct"] - 100 * (1 - 82 / 8192)) < 1e-9
    assert abs(ctx["wire_ms_at_link"] - 2 * 65536 * 82 * 2 / 1e4) < 1e-6      # 80 Mbps = 1e4 B/ms
