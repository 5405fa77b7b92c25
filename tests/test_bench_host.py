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
    rf = bench.roofline(tr, N, HD, 1, 1724.3, "bf16 sustained, measured", "no-such-variant", 6678.5, V=V)
    assert rf["kernel"] == "dh_gemm" and rf["bound"] == "tensor" and rf["launches_per_step"] == 10
    want = 2.0 * N * HD * (V / 10) / (1.47e-3) / 1e12        # algorithmic flops of a mean launch / its time
    assert rf["achieved"] == pytest.approx(want, rel=1e-3)
    assert rf["frac"] == pytest.approx(want / 1724.3, rel=1e-3)
    assert sum(rf["time_share"].values()) == pytest.approx(1.0, abs=1e-3)
    assert rf["traffic"] is None                              # nothing stored for this variant
    z = rf["dz_logits_hbm"]                                   # fp32 logits in, bf16 dZ out: 6 bytes a column
    assert z["bytes_per_launch"] == pytest.approx(6.0 * N * V / 10, rel=1e-9)
    assert z["achieved"] == pytest.approx(6.0 * N * V / 10 / 0.29e-3 / 1e9, rel=1e-3)
    assert z["frac"] == pytest.approx(z["achieved"] / 6678.5, rel=1e-3)


def test_decode_launch_below_the_ridge_is_hbm_bound():
    """A sampling GEMM over 256 rows reads the 1.27 GB head for 0.3 PFLOP: its
    bound is HBM, its algorithmic bytes the head plus the gathered rows."""
    tr = [(K("compact"), 0, 0.02), (K("sample_gemm"), V, 0.234), (K("logp_merge"), 0, 0.05)]
    rf = bench.roofline(tr, 256, HD, 1, 1724.3, "bf16 sustained, measured", "x", 6678.5, V=V)
    assert rf["bound"] == "hbm" and rf["unit"] == "GB/s"
    alg = 2.0 * HD * V + 2.0 * HD * 256
    assert rf["bytes_per_launch"] == pytest.approx(alg)
    assert rf["achieved"] == pytest.approx(alg / 0.234e-3 / 1e9, rel=1e-3)
    # the same launch over 19,572 rows is far above the ridge: tensor-bound
    tr = [(K("sample_gemm"), V, 16.0)]
    assert bench.roofline(tr, N, HD, 1, 1724.3, "x", "x", 6678.5, V=V)["bound"] == "tensor"


def test_top_p_selection_figure():
    tr = [(K("sample_gemm"), V, 1.6), (K("top_p"), V, 0.65)]
    rf = bench.roofline(tr, 2048, HD, 1, 1724.3, "x", "x", 6678.5, V=V)
    t = rf["top_p_hbm"]                                       # the stored logits read once
    assert t["bytes_per_launch"] == pytest.approx(4.0 * 2048 * V)
    assert t["achieved"] == pytest.approx(4.0 * 2048 * V / 0.65e-3 / 1e9, rel=1e-3)


def test_stored_traffic_is_scaled_to_the_launch_and_keyed_by_source(tmp_path):
    """traffic.txt lines count only for the current kernel sources, the same
    path variant, and a capture on the same hidden size and vocabulary; a
    line's bytes scale with the rows of the bench batch over the capture's and
    with the vocabulary columns of the launch over the capture's."""
    tr = _step_trace()
    kh = bench.kernel_hash()
    path = tmp_path / "traffic.txt"
    path.write_text("# comment line\n"
                    f"{kh} fwdbwd+kept fwdbwd_mid 5000 dh_gemm 1000000000 16384\n"
                    f"{kh} fwdbwd fwdbwd_mid 5000 dh_gemm 2000000000 16384\n"
                    f"{kh} fwdbwd fwdbwd_small 5931 dw_gemm 7 16384\n"          # another vocabulary: not used
                    f"0000000000000000 fwdbwd fwdbwd_mid 5000 dw_gemm 5 16384\n")  # older sources: not used
    got = bench.stored_traffic("fwdbwd", "dh_gemm", HD, V, N, path=str(path))
    assert got is not None and got[1] == 16384
    assert got[0] == pytest.approx(2e9 * N / 5000, rel=1e-12)
    rf = bench.roofline(tr, N, HD, 1, 1724.3, "x", "fwdbwd+kept", 6678.5, V=V, traffic_path=str(path))
    assert rf["kernel"] == "dh_gemm"
    assert rf["traffic"] == pytest.approx(1e9 * N / 5000 * (V / 10) / 16384, rel=1e-9)
    assert "fwdbwd_mid" in rf["traffic_from"]
    assert bench.stored_traffic("fwdbwd", "dw_gemm", HD, V, N, path=str(path)) is None
    assert bench.stored_traffic("fwdbwd", "no_such_kernel", HD, V, N, path=str(path)) is None
    # the committed file: every line well-formed, each capture a workload of a few GB on the device
    for line in open(bench.TRAFFIC_PATH):
        if line.startswith("#") or not line.strip():
            continue
        f = line.split()
        assert len(f) == 7 and f[2] in bench.wl.ALL_WORKLOADS, line
        cw = bench.wl.ALL_WORKLOADS[f[2]]
        assert cw.T <= 16384, "captures beyond the launch list stay on small cases"


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
