"""Shared helpers for the tests: tolerances of the parity bar and tensor plumbing."""
from __future__ import annotations

import numpy as np

# Parity bar (absolute log-prob error, relative loss error, relative Frobenius
# error of the gradients); advantages and masks are compared bit for bit.
LOGP_ATOL = 2e-3
LOSS_RTOL = 1e-3
GRAD_RTOL = 1e-2


# Within the log-prob tolerance, the ratio rho = exp(logp - old) of a token
# closer than this to a clip boundary 1 -+ clip_eps can fall on either side of
# it on the GPU (fp32) and in the oracle (fp64), and the min() of Eq. 1 then
# takes different branches: the token's gradient is not unique there (the
# loss is continuous, so it is unaffected).
RHO_MARGIN = 5e-3


def clear_of_clip_kink(logp, old, clip_eps: float, margin: float = RHO_MARGIN, step: float = 0.02):
    """The old log-probs with every token's rho moved at least `margin` away from
    both clip boundaries: a token that is too close gets its old log-prob
    shifted by `step` (rho scaled by e^step) away from the boundary.  Parity
    inputs use this so that the gradient they compare is unique."""
    lp = np.asarray(logp, dtype=np.float64)
    o = np.asarray(old)
    out = o.astype(np.float64).copy()
    rho = np.exp(lp - out)
    for b in (1.0 - clip_eps, 1.0 + clip_eps):
        near = np.abs(rho - b) < margin
        out[near] -= step * np.where(rho[near] >= b, 1.0, -1.0)
    return out.astype(o.dtype)


def near_clip_kink(logp, old, clip_eps: float, margin: float = RHO_MARGIN):
    """Mask of the tokens whose rho lies within `margin` of a clip boundary."""
    rho = np.exp(np.asarray(logp, dtype=np.float64) - np.asarray(old, dtype=np.float64))
    return (np.abs(rho - (1.0 - clip_eps)) < margin) | (np.abs(rho - (1.0 + clip_eps)) < margin)


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
