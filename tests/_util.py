"""Shared helpers for the tests: tolerances of the parity bar and tensor plumbing."""
from __future__ import annotations

import numpy as np

# Parity bar (absolute log-prob error, relative loss error, relative Frobenius
# error of the gradients); advantages and masks are compared bit for bit.
LOGP_ATOL = 2e-3
LOSS_RTOL = 1e-3
GRAD_RTOL = 1e-2


def loss_scale(loss_ref: float, w, ell) -> float:
    """Denominator of the loss check: |loss| or, when the advantages cancel and
    the loss sits near 0, the size of the terms it sums (sum_t |w_t l_t|)."""
    return max(abs(loss_ref), float(np.sum(np.abs(np.asarray(w) * np.asarray(ell)))))


def rel_fro(got, want) -> float:
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    den = np.linalg.norm(want)
    return float(np.linalg.norm(got - want) / den) if den > 0 else float(np.linalg.norm(got))


def dev_tensor(a, dtype, device="cuda"):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).view(dtype).to(device)
