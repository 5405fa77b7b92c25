"""Host logic of bench.py on CPU: the roofline of the dominant kernel from a
launch trace, the HBM figures of the element-wise passes, and the lookup of
stored DRAM traffic.  (The device-timed run itself needs a GPU.)"""
import json
import os
import subprocess
import sys

import pytest

import bench

N, HD, V = 19572, 4096, 155136
K = bench.KIND_NAMES.index


def _step_trace(dh_ms=1.47):
    """One step of the kept-logits backward: forward, ten chunks of dZ pass + dH + dW."""
    tr = [(K("compact"), 0, 0.05), (K("lse_gemm"), V, 14.5), (K("loss"), 0, 0.03)]
    for c in range(10):
        cols = 16384 if c < 9 else V - 9 * 16384
        tr += [(K("dz_logits"), cols, 0.29), (K("dh_gemm"), cols, dh_ms), (K("dw_gemm"), cols, 1.43)]
    return tr


def test_dominant_kernel_achieved_rate_and_shares():
    tr = _step_trace()
    rf = bench.roofline(tr, N, HD, 1, 1724.3, "bf16 sustained, measured", "no-such-workload", 6678.5)
    assert rf["kernel"] == "dh_gemm" and rf["bound"] == "tensor" and rf["launches_per_step"] == 10
    want = 2.0 * N * HD * (V / 10) / (1.47e-3) / 1e12        # algorithmic flops of a mean launch / its time
    assert rf["achieved"] == pytest.approx(want, rel=1e-3)
    assert rf["frac"] == pytest.approx(want / 1724.3, rel=1e-3)
    assert sum(rf["time_share"].values()) == pytest.approx(1.0, abs=1e-3)
    assert rf["traffic"] is None                              # nothing stored for this workload name
    z = rf["dz_logits_hbm"]                                   # fp32 logits in, bf16 dZ out: 6 bytes a column
    assert z["bytes_per_launch"] == pytest.approx(6.0 * N * V / 10, rel=1e-9)
    assert z["achieved"] == pytest.approx(6.0 * N * V / 10 / 0.29e-3 / 1e9, rel=1e-3)
    assert z["frac"] == pytest.approx(z["achieved"] / 6678.5, rel=1e-3)


def test_decode_launch_below_the_ridge_is_hbm_bound():
    """A sampling GEMM over 256 rows reads the 1.27 GB head for 0.3 PFLOP: its
    bound is HBM, its algorithmic bytes the head plus the gathered rows."""
    tr = [(K("compact"), 0, 0.02), (K("sample_gemm"), V, 0.234), (K("logp_merge"), 0, 0.05)]
    rf = bench.roofline(tr, 256, HD, 1, 1724.3, "bf16 sustained, measured", "x", 6678.5)
    assert rf["bound"] == "hbm" and rf["unit"] == "GB/s"
    alg = 2.0 * HD * V + 2.0 * HD * 256
    assert rf["bytes_per_launch"] == pytest.approx(alg)
    assert rf["achieved"] == pytest.approx(alg / 0.234e-3 / 1e9, rel=1e-3)
    # the same launch over 19,572 rows is far above the ridge: tensor-bound
    tr = [(K("sample_gemm"), V, 16.0)]
    assert bench.roofline(tr, N, HD, 1, 1724.3, "x", "x", 6678.5)["bound"] == "tensor"


def test_top_p_selection_figure():
    tr = [(K("sample_gemm"), V, 1.6), (K("top_p"), V, 0.65)]
    rf = bench.roofline(tr, 2048, HD, 1, 1724.3, "x", "x", 6678.5)
    t = rf["top_p_hbm"]                                       # the stored logits read once
    assert t["bytes_per_launch"] == pytest.approx(4.0 * 2048 * V)
    assert t["achieved"] == pytest.approx(4.0 * 2048 * V / 0.65e-3 / 1e9, rel=1e-3)


def test_stored_traffic_is_scaled_to_the_launch_and_keyed_by_source():
    """traffic.txt lines count only for the current kernel sources; a line's
    bytes scale with the vocabulary columns of the launch."""
    tr = _step_trace()
    line = bench.stored_traffic("fwdbwd_8b", "dh_gemm")
    if line is None:
        pytest.skip("no traffic line for the current kernel sources")
    bytes_ref, cols_ref = line
    rf = bench.roofline(tr, N, HD, 1, 1724.3, "x", "fwdbwd_8b", 6678.5)
    assert rf["traffic"] == pytest.approx(bytes_ref * (V / 10) / cols_ref, rel=1e-9)
    assert bench.stored_traffic("fwdbwd_8b", "no_such_kernel") is None


def test_reference_arm_prints_one_contract_line():
    """bench.py --impl reference: the float64 oracle on the host cores prints
    one JSON line with the contract's keys on rank 0; another rank prints
    nothing and exits 0."""
    cmd = [sys.executable, os.path.join(bench.ROOT, "bench.py"), "--impl", "reference", "--workload", "tiny_fwdbwd",
           "--steps", "2", "--warmup", "1", "--cpu-sample-tokens", "64"]
    env = {k: v for k, v in os.environ.items() if k not in ("RANK", "WORLD_SIZE", "LOCAL_RANK")}
    out = subprocess.run(cmd, capture_output=True, text=True, timeout=300, cwd=bench.ROOT, env=env)
    assert out.returncode == 0, out.stderr
    lines = [ln for ln in out.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC and d["unit"] == "tokens/s"
    assert d["value"] > 0 and d["steps"] == 2 and d["warmup"] == 1 and d["higher_is_better"] is True
    assert d["dtype"] == "f64" and d["config"]["workload"] == "tiny_fwdbwd"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["cores"] >= 1 and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    out = subprocess.run(cmd, capture_output=True, text=True, timeout=300, cwd=bench.ROOT, env=dict(env, RANK="1"))
    assert out.returncode == 0, out.stderr
    assert not [ln for ln in out.stdout.splitlines() if ln.startswith("{")]
