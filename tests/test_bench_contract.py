"""bench.py's output contract: one JSON line with the keys the driver reads.
The reference arm (the oracle on host cores) runs on CPU; the GPU arm on a
GPU machine."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run(args, timeout):
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], cwd=ROOT,
                       capture_output=True, text=True, timeout=timeout)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout
    return json.loads(lines[0])


def test_reference_arm_line():
    d = _run(["--impl", "reference", "--workload", "tiny_f32", "--steps", "1", "--warmup", "3"],
             timeout=600)
    assert d["impl"] == "reference"
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "higher_is_better",
              "config", "cpu_baseline", "e2e"):
        assert k in d, k
    assert d["value"] > 0 and d["higher_is_better"] is False
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["value"] == d["value"]


def test_warmup_below_three_is_refused():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--warmup", "1"],
                       cwd=ROOT, capture_output=True, text=True, timeout=120)
    assert r.returncode != 0


@pytest.mark.gpu
def test_gpu_arm_line():
    d = _run(["--steps", "20", "--warmup", "3", "--skip-cpu"], timeout=600)
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
              "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config", "roofline",
              "e2e", "clocks", "gpu_launches"):
        assert k in d, k
    assert d["n_gpus"] == 1 and d["steps"] == 20 and d["warmup"] == 3
    assert d["config"]["workload"] == "llama8b_k16"
    rf = d["roofline"]
    assert rf["bound"] == "hbm" and 0 < rf["frac"] < 1.2 and rf["peak"] > 0
    assert abs(rf["frac"] - rf["achieved"] / rf["peak"]) < 1e-3
    e2e = d["e2e"]
    assert e2e["value"] >= d["value"] * 0.99 and e2e["h2d_bytes_per_step"] > 0
    assert d["gpu_launches"] > 0
    assert "sm_mhz" in d["clocks"] and "reasons" in d["clocks"]


def test_algorithmic_bytes_at_llama_shapes():
    """The roofline's byte count at the Llama-3.1-8B workload, written out
    from its shapes (B = 1, k = 16 with 15 masked rows, 32/8 heads of 128,
    cache 4096, hidden 4096, vocabulary 128256, bf16)."""
    import numpy as np

    import bench
    import gen
    w = gen.get_workload("llama8b_k16")
    assert (w.batch, w.block_k, w.n_q_heads, w.n_kv_heads, w.head_dim) == (1, 16, 32, 8, 128)
    assert (w.hidden, w.vocab, w.dtype) == (4096, 128256, "bf16")
    masked = np.ones((1, 16), dtype=np.uint8)
    masked[0, 0] = 0
    ab = bench.algorithmic_bytes(w, {"cache_len": np.array([4096], np.int32), "masked": masked})
    # K and V cache rows 2*4096*8*128*2 = 16,777,216; block K/V 2*16*8*128*2 =
    # 65,536; Q and O 2*16*32*128*2 = 262,144; the cache length 4
    assert ab["attention"] == 16_777_216 + 65_536 + 262_144 + 4
    # W 128256*4096*2 = 1,050,673,152; 15 hidden rows 15*4096*2 = 122,880;
    # 15 Gumbel rows 15*128256*4 = 7,695,360; masked flags, entropies and
    # tokens 16*(1+4+4) = 144
    assert ab["head"] == 1_050_673_152 + 122_880 + 7_695_360 + 144
    assert ab["R"] == 15
    # with the noise drawn in the kernel, the Gumbel rows are not read
    ab_p = bench.algorithmic_bytes(w, {"cache_len": np.array([4096], np.int32), "masked": masked},
                                   noise="philox")
    assert ab["head"] - ab_p["head"] == 7_695_360
