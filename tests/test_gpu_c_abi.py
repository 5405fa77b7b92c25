"""The C ABI driven from a plain C11 program on the GPU (tests/c_abi_check.c):
device memory from cudaMalloc, Eq. 2 advantages and log-probs through
libgrpo.so, no Python on the path.  Its printed results must match the float64
oracle on the inputs it prints: advantages bit for bit, log-probs within 2e-3."""
import subprocess

import numpy as np
import pytest

import oracle
from tests._util import LOGP_ATOL
from tests.test_abi import _build_c_check

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2507_05687_gb300 import build as build_mod  # noqa: E402

build_mod.build()


def test_c_program_matches_the_oracle(tmp_path):
    exe = _build_c_check(tmp_path)
    out = subprocess.run([exe, "device"], capture_output=True, text=True, timeout=120)
    assert out.returncode == 0, out.stdout[-2000:] + out.stderr
    vals = {"adv": [], "logp": [], "H": [], "W": [], "y": []}
    for line in out.stdout.splitlines():
        key, *rest = line.split()
        vals[key].append(rest)
    adv = np.array([float(v[0]) for v in vals["adv"]], dtype=np.float32)
    logp = np.array([float(v[0]) for v in vals["logp"]])
    T, HD, V, G = len(logp), 64, 300, 4
    H = np.array([int(v[0]) for v in vals["H"]], dtype=np.uint16).reshape(T, HD)
    W = np.array([int(v[0]) for v in vals["W"]], dtype=np.uint16).reshape(V, HD)
    y = np.array([int(v[0]) for v in vals["y"]])
    m = np.array([int(v[1]) for v in vals["y"]], dtype=np.uint8)
    rewards = np.array([0, 1, 0.5, 0, 1, 1, 0, 0.5], dtype=np.float32)
    want_adv = oracle.group_advantages(rewards, G, float(np.float32(1e-6)))
    assert np.array_equal(adv.view(np.uint32), want_adv.view(np.uint32))
    want, _ = oracle.token_logprobs(H, W, y, m)
    assert np.all(logp[m == 0] == 0.0)
    assert np.abs(logp - want).max() <= LOGP_ATOL
