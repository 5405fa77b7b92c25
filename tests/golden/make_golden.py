"""Write the float64 oracle's log-probs for the 8B-shaped workloads.

    python tests/golden/make_golden.py [batch8b] [long_8b] [ragged_8b]

Calls only oracle/ and the seeded generators of workloads.py.  For each batch
it stores, in compacted order (unmasked rows by increasing position):

* lse_policy  float64  log-sum-exp of H_t W^T under the policy head
* old_logp    float32  the oracle's log pi_old(y_t), rounded once to float32
* ref_logp    float32  the oracle's log pi_ref(y_t), rounded once to float32
* checksums of the regenerated inputs, so a test on another host can confirm
  it rebuilt the same arrays before comparing against these values.

old_logp / ref_logp are inputs of the loss (they come from earlier forward
passes of the old and reference policies); lse_policy is an expected value.
A full run takes about an hour of float64 BLAS on 8 cores.
"""
from __future__ import annotations

import os
import sys
import time

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import oracle  # noqa: E402
import workloads as wl  # noqa: E402

BATCHES = {"batch8b": "fwdbwd_8b", "long_8b": "long_8b", "ragged_8b": "ragged_8b"}


def checksums(w, H, W, y, mask):
    idx = wl.valid_index(mask)
    return {
        "ck_h": np.uint64(H[idx].astype(np.uint64).sum()),
        "ck_w": np.uint64(W.astype(np.uint64).sum()),
        "ck_y": np.uint64(y[idx].astype(np.uint64).sum()),
        "n_valid": np.int64(idx.size),
    }


def make(batch: str) -> str:
    w = wl.WORKLOADS[BATCHES[batch]]
    t0 = time.time()
    H = wl.gen_hidden(w)
    y = wl.gen_targets(w)
    mask = wl.gen_mask(w)
    W = wl.gen_weight(w, "policy")
    idx = wl.valid_index(mask)
    print(f"[{batch}] inputs {time.time() - t0:.1f}s  N_valid={idx.size}", flush=True)
    out = checksums(w, H, W, y, mask)
    _, lse = oracle.token_logprobs(H, W, y, mask)
    out["lse_policy"] = lse[idx]
    print(f"[{batch}] policy pass {time.time() - t0:.1f}s", flush=True)
    for which in ("old", "ref"):
        Wx = wl.gen_weight(w, which, policy=W)
        lp, _ = oracle.token_logprobs(H, Wx, y, mask)
        out[f"{which}_logp"] = lp[idx].astype(np.float32)
        del Wx
        print(f"[{batch}] {which} pass {time.time() - t0:.1f}s", flush=True)
    path = os.path.join(HERE, f"{batch}.npz")
    np.savez(path, **out)
    print(f"[{batch}] wrote {path} in {time.time() - t0:.1f}s", flush=True)
    return path


if __name__ == "__main__":
    for b in (sys.argv[1:] or list(BATCHES)):
        make(b)
