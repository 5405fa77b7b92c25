"""Pure-Python brute force of the same definitions, for tiny shapes (test infrastructure).

No vectorisation, no max shift in the log-sum-exp, no chunking: each quantity
is the sum written out with explicit loops, so it can be read against Eq. 1
and Eq. 2 of Section 3.3 term by term.  Only for T, Hd, V of a few dozen.
"""
from __future__ import annotations

import math


def advantages(rewards, G, eps=1e-6):
    """Eq. 2 with the sample standard deviation (divide by G - 1)."""
    out = []
    for g0 in range(0, len(rewards), G):
        grp = [float(r) for r in rewards[g0:g0 + G]]
        mu = sum(grp) / G
        var = sum((r - mu) ** 2 for r in grp) / (G - 1)
        sd = math.sqrt(var)
        out.extend((r - mu) / (sd + eps) for r in grp)
    return out


def logprobs(H, W, targets, mask):
    """log( exp(z_{t,y}) / sum_v exp(z_{t,v}) ) with z_{t,v} = sum_k H[t][k] W[v][k]."""
    T, V, Hd = len(H), len(W), len(H[0])
    out = []
    for t in range(T):
        if not mask[t]:
            out.append(0.0)
            continue
        z = [sum(H[t][k] * W[v][k] for k in range(Hd)) for v in range(V)]
        total = sum(math.exp(zv) for zv in z)
        out.append(z[targets[t]] - math.log(total))
    return out


def loss(logp, old, ref, adv, mask, n_resp, L, clip_eps, beta, agg_mode=0, kl_clamp=math.inf):
    """Negated Eq. 1; agg_mode 0 = masked token-mean, 1 = per-response mean then mean.
    kl_clamp caps each token's KL value (no cap by default)."""
    total_tok = sum(1 for t in range(n_resp * L) if mask[t])
    acc = 0.0
    for i in range(n_resp):
        n_i = sum(1 for j in range(L) if mask[i * L + j])
        for j in range(L):
            t = i * L + j
            if not mask[t]:
                continue
            rho = math.exp(logp[t] - old[t])
            A = adv[i]
            clipped = min(max(rho, 1.0 - clip_eps), 1.0 + clip_eps)
            s = min(rho * A, clipped * A)
            kl = math.exp(ref[t] - logp[t]) - (ref[t] - logp[t]) - 1.0
            if kl > kl_clamp:
                kl = kl_clamp
            ell = -(s - beta * kl)
            if agg_mode == 0:
                acc += ell / total_tok
            else:
                acc += ell / (n_resp * n_i)
    return acc
