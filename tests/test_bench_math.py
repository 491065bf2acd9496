"""The measurement arithmetic of bench.py (CPU): the algorithmic work per step and per vocabulary
launch that the roofline fractions divide by, checked against the per-configuration figures
computed from the model shapes (GFLOP, weight and activation MB), and the choice of the bound."""
import pytest

import bench
from paper_2605_29707_gb300 import inputs

# config -> (GFLOP per step, weight MB, activation MB), MB = 1e6 bytes, from the shapes alone:
# FLOPs = 2 M (H V + r V + 3 d_s H + 3 d_s^2 + (H + d_s) r); weights = every matrix once in bf16;
# activations = hidden + gathered embedding rows (bf16) + ids (int32)
SHAPES = {
    "tiny": (0.051, 12.7, 0.004),
    "qwen3-1.7b": (11.53, 720.6, 0.13),
    "qwen3-8b": (21.70, 1356.5, 0.26),
    "qwen3-8b-b32": (694.5, 1356.5, 8.4),
    "qwen3-32b-b64": (1714.7, 1674.5, 21.0),
}


@pytest.mark.parametrize("name", list(SHAPES))
def test_step_work_matches_the_shapes(name):
    c = inputs.CONFIGS[name]
    gflop, w_mb, a_mb = SHAPES[name]
    w = bench.step_work(c)
    assert w["flops"] / 1e9 == pytest.approx(gflop, rel=2e-3, abs=1e-3)
    # the figures are printed to 0.1 MB (weights) and 2-3 digits (activations)
    assert w["bytes"] / 1e6 == pytest.approx(w_mb + a_mb, abs=0.06)


def test_vocab_launch_bytes_at_the_8b_shape():
    """W_lm + W2 once, hidden + u, and the 16 x 149 partial records of 8-entry lists."""
    c = inputs.CONFIGS["qwen3-8b"]
    w = bench.vocab_work(c, 152)
    assert w["plan"]["nchunks"] == 149 and w["plan"]["rec_words"] == 18 and w["plan"]["swap"]
    assert w["bytes"] == 151936 * 4352 * 2 + 16 * 4352 * 2 + 16 * 149 * 18 * 4 == 1322761856
    assert w["per_unit_bytes"] * w["units"] == 151936 * 4352 * 2


def test_roofline_takes_the_slower_of_memory_and_tensor_time():
    peaks = {"hbm_gbs": 6000.0, "bf16_tflops": 2000.0, "bf16_tflops_sustained": 1500.0, "source": "test"}
    # 6 GB in 1 ms at 6000 GB/s: memory-bound, frac 1.0
    r = bench.roofline_entry(6e9, 1e12, 1.0, peaks, sustained=False)
    assert r["bound"] == "hbm" and r["frac"] == pytest.approx(1.0) and r["unit"] == "GB/s"
    # 3 PFLOP in 2 s against the sustained 1500 TFLOP/s: tensor-bound, frac 1.0
    r = bench.roofline_entry(1e6, 3e15, 2000.0, peaks, sustained=True)
    assert r["bound"] == "tensor" and r["frac"] == pytest.approx(1.0) and r["unit"] == "TFLOP/s"


def test_multi_gpu_launch_is_refused_without_running():
    """The library is single-GPU (its vocabulary GEMM multicasts weight tiles within a cluster,
    which only 1-GPU runs may use): a torchrun launch or --gpus > 1 prints one 'unavailable' line
    from rank 0, the other ranks print nothing, and nothing runs."""
    import json
    import os
    import subprocess
    import sys

    assert bench.single_gpu_refusal(1, 1) is None
    line = bench.single_gpu_refusal(2, 1)
    assert line["unavailable"] and line["n_gpus"] == 2
    assert bench.single_gpu_refusal(1, 4)["n_gpus"] == 4
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    for rank, expect in (("0", True), ("1", False)):
        env = dict(os.environ, WORLD_SIZE="2", RANK=rank, LOCAL_RANK=rank)
        r = subprocess.run([sys.executable, os.path.join(root, "bench.py"), "--gpus", "2", "--steps", "3"],
                           env=env, capture_output=True, text=True, timeout=120)
        assert r.returncode == 0, r.stderr
        out = [ln for ln in r.stdout.splitlines() if ln.strip()]
        if expect:
            assert len(out) == 1 and json.loads(out[0])["unavailable"] == bench.SINGLE_GPU
        else:
            assert out == []
