"""Write the float64 oracle's log-probs for the 8B-shaped workloads.

    python tests/golden/make_golden.py [batch8b] [long_8b] [ragged_8b]
    python tests/golden/make_golden.py loss [batch8b] [long_8b] [ragged_8b]

Calls only oracle/ and the seeded generators of workloads.py.  For each batch
it stores, in compacted order (unmasked rows by increasing position):

* lse_policy  float64  log-sum-exp of H_t W^T under the policy head
* old_logp    float32  the oracle's log pi_old(y_t), rounded once to float32
* ref_logp    float32  the oracle's log pi_ref(y_t), rounded once to float32
* checksums of the regenerated inputs, so a test on another host can confirm
  it rebuilt the same arrays before comparing against these values.

old_logp / ref_logp are inputs of the loss (they come from earlier forward
passes of the old and reference policies); lse_policy is an expected value.
A full run takes about an hour of float64 BLAS on 8 cores.  The `loss` mode
reads those files back and writes <batch>_loss.json, the oracle's loss of
each batch (see make_loss), in a minute or two.
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


def make_loss(batch: str) -> str:
    """<batch>_loss.json: the oracle's loss of the batch in both aggregations
    (Eq. 1 as a masked token-mean, agg_mode 0, and as printed, agg_mode 1) and
    the size of the terms it sums (sum_t |w_t l_t|), from the log-sum-exps
    and old / reference log-probs stored in <batch>.npz, the advantages of
    the batch's rewards (Eq. 2) and the float64 target logits."""
    import json
    w = wl.WORKLOADS[BATCHES[batch]]
    d = np.load(os.path.join(HERE, f"{batch}.npz"))
    H, W, y, mask = wl.gen_hidden(w), wl.gen_weight(w, "policy"), wl.gen_targets(w), wl.gen_mask(w)
    ck = checksums(w, H, W, y, mask)
    for k in ("ck_h", "ck_w", "ck_y", "n_valid"):
        assert ck[k] == d[k], k
    idx = wl.valid_index(mask)
    logp = np.zeros(w.T)
    logp[idx] = oracle.target_logits(H, W, y, idx) - d["lse_policy"]
    old = np.zeros(w.T, np.float32)
    ref = np.zeros(w.T, np.float32)
    old[idx], ref[idx] = d["old_logp"], d["ref_logp"]
    adv = oracle.group_advantages(wl.gen_rewards(w), w.G, float(np.float32(w.adv_eps)))
    out = {"workload": w.name, "n_valid": int(idx.size), "clip_eps": w.clip_eps, "beta": w.beta}
    for agg in (0, 1):
        loss, _, tt = oracle.grpo_loss(logp, old, ref, adv, mask, w.n_resp, w.L, w.clip_eps, w.beta, agg)
        out[f"loss_agg{agg}"] = loss
        out[f"sum_abs_terms_agg{agg}"] = float(np.sum(np.abs(tt["w"] * tt["ell"])))
    path = os.path.join(HERE, f"{batch}_loss.json")
    with open(path, "w") as f:
        json.dump(out, f, indent=1)
        f.write("\n")
    print(f"[{batch}] wrote {path}", flush=True)
    return path


if __name__ == "__main__":
    args = sys.argv[1:]
    if args[:1] == ["loss"]:
        for b in (args[1:] or list(BATCHES)):
            make_loss(b)
    else:
        for b in (args or list(BATCHES)):
            make(b)
