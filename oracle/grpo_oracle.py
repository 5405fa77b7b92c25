"""Float64 CPU oracle of the GRPO hot path (test infrastructure).

Test infrastructure only: ``tests/``, ``__graft_entry__.smoke()`` and the CPU
baseline leg of ``bench.py`` may import it; the library never does and shares
no code with it.

What it computes, in the paper's notation (Section 3.3):

* Eq. 2, the group-relative advantage
      A_i = (r_i - mean_j r_j) / (std_j r_j + eps)
  over the G responses of one prompt (readings: the N of Eq. 2 is the group
  size G; std is the sample std, ddof = 1; eps = 1e-6 keeps a zero-std group
  at A = 0), broadcast to every token of response i.
* pi_theta(o_{i,t} | q, o_{i,<t}) inside Eq. 1: the log-softmax of the LM-head
  logits z_t = H_t W^T (temperature 1), taken at the sampled token y_t.
* the braces of Eq. 1 per token:  rho = pi_theta / pi_old = exp(logp - old),
      s = min(rho A, clip(rho, 1-eps_c, 1+eps_c) A)
      KL = exp(ref - logp) - (ref - logp) - 1     (per-token k3 estimator of
           D_KL(pi_theta || pi_ref) from the GRPO paper the method cites)
      l = -(s - beta KL)                          (loss = -J)
  Optionally the KL value is capped, KL = min(k3, kl_clamp) (the paper does
  not fix the estimator; a cap bounds one token's penalty when the reference
  and the policy disagree strongly).  A capped token has no KL gradient.
* the aggregation of Eq. 1: agg_mode 1 is Eq. 1 as printed,
      (1/n_resp) sum_i (1/|o_i|) sum_t l_{i,t};
  agg_mode 0 (default) is the masked token-mean sum_t mask_t l_t / N_valid.
* the gradient of that loss to H and W: with g_t = dloss/dlogp_t,
      dZ_{t,v} = g_t (1[v = y_t] - p_{t,v}),  dH = dZ W,  dW = dZ^T H.
  At the kink of min() (rho A == clip(rho) A) the unclipped branch is taken.

* the rollout draw that produces o_{i,t} ~ pi_theta_old (the sampling step
  before Eq. 1, Section 3.3): Gumbel-max over softmax(z_t / temperature) with
  Philox4x32-10 noise, optionally restricted to the nucleus (top-p) of that
  distribution (Holtzman et al., "The Curious Case of Neural Text
  Degeneration", 2020): the smallest set of the most probable tokens whose
  mass reaches top_p, every token tied with its least probable member
  included.  Gumbel-max over a subset draws from the distribution
  renormalised on that subset.

Rows with mask 0 have logp = 0, weight 0, and zero dH rows.
Every floating value is float64; bf16 inputs are widened exactly.
"""
from __future__ import annotations

import numpy as np

# ---------------------------------------------------------------------------
# inputs
# ---------------------------------------------------------------------------


def widen_bf16(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) -> float64, exactly (a bf16 is the top half of an f32)."""
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


def as_f64(x) -> np.ndarray:
    """Float64 view of a float array, or exact widening of bf16 bits given as uint16."""
    x = np.asarray(x)
    if x.dtype == np.uint16:
        return widen_bf16(x)
    return np.asarray(x, dtype=np.float64)


# ---------------------------------------------------------------------------
# Eq. 2: group-relative advantage
# ---------------------------------------------------------------------------


def group_advantages(rewards, G: int, eps: float = 1e-6, ddof: int = 1) -> np.ndarray:
    """Eq. 2 per group of G consecutive responses; float64 math, rounded once to float32."""
    r = np.asarray(rewards, dtype=np.float64)
    if G < 2 or r.size % G:
        raise ValueError("need G >= 2 and n_resp % G == 0")
    g = r.reshape(-1, G)
    mu = g.mean(axis=1, keepdims=True)
    sd = g.std(axis=1, ddof=ddof, keepdims=True)
    return ((g - mu) / (sd + eps)).reshape(-1).astype(np.float32)


# ---------------------------------------------------------------------------
# pi_theta(o_t | ...): log-softmax over the vocabulary at the sampled token
# ---------------------------------------------------------------------------


def token_logprobs(H, W, targets, mask, vocab_chunk: int = 8192, row_chunk: int = 4096):
    """log softmax(H_t W^T)[y_t] for unmasked rows.

    Returns (logp [T], lse [T]) in float64; masked rows are 0.  The logits are
    formed chunk by chunk over the vocabulary, with a running max and a running
    sum of exp(z - max) per row, so the [T, V] matrix is never held at once.
    """
    H = np.asarray(H)
    W = as_f64(W)
    y = np.asarray(targets, dtype=np.int64)
    m = np.asarray(mask) != 0
    T, V = H.shape[0], W.shape[0]
    logp = np.zeros(T, dtype=np.float64)
    lse = np.zeros(T, dtype=np.float64)
    idx = np.flatnonzero(m)
    for r0 in range(0, idx.size, row_chunk):
        rows = idx[r0:r0 + row_chunk]
        Hr = as_f64(H[rows])
        yr = y[rows]
        run_max = np.full(rows.size, -np.inf)
        run_sum = np.zeros(rows.size)
        zy = np.zeros(rows.size)
        for v0 in range(0, V, vocab_chunk):
            v1 = min(V, v0 + vocab_chunk)
            Z = Hr @ W[v0:v1].T
            new_max = np.maximum(run_max, Z.max(axis=1))
            run_sum = run_sum * np.exp(run_max - new_max) + np.exp(Z - new_max[:, None]).sum(axis=1)
            run_max = new_max
            hit = (yr >= v0) & (yr < v1)
            zy[hit] = Z[np.flatnonzero(hit), yr[hit] - v0]
        l = run_max + np.log(run_sum)
        lse[rows] = l
        logp[rows] = zy - l
    return logp, lse


def target_logits(H, W, targets, rows, row_chunk: int = 16384) -> np.ndarray:
    """z_{t, y_t} = H_t . W_{y_t} in float64 for the listed rows: the logit of
    the sampled token, from which logp_t = z_{t, y_t} - LSE_t (Eq. 1's
    pi_theta at o_{i,t}) once the row's log-sum-exp is known."""
    rows = np.asarray(rows, dtype=np.int64)
    y = np.asarray(targets, dtype=np.int64)
    Hs, Ws = np.asarray(H), np.asarray(W)
    out = np.empty(rows.size)
    for a in range(0, rows.size, row_chunk):
        r = rows[a:a + row_chunk]
        out[a:a + r.size] = np.einsum("ij,ij->i", as_f64(Hs[r]), as_f64(Ws[y[r]]))
    return out


# ---------------------------------------------------------------------------
# Eq. 1: per-token terms, weights, loss and its derivative in logp
# ---------------------------------------------------------------------------


def token_advantages(adv, n_resp: int, L: int) -> np.ndarray:
    """A_{i,t} = A_i for every padded row of response i (Eq. 2 broadcast)."""
    a = np.asarray(adv, dtype=np.float64)
    assert a.size == n_resp
    return np.repeat(a, L)


def token_terms(logp, old_logp, ref_logp, adv_tok, clip_eps: float, beta: float, kl_clamp: float = np.inf):
    """The braces of Eq. 1 for every row.

    Returns a dict with rho, the clipped-surrogate value s, the k3 KL, the
    per-token loss l = -s + beta KL and the 0/1 flag 'unclipped' (the min()
    picks rho A; ties count as unclipped).

    kl_clamp caps the per-token KL value: KL = min(k3, kl_clamp), and a token
    whose k3 lies above the cap contributes a constant (no KL gradient); a tie
    counts as inside.  The default (infinity) is the plain k3 estimator.  The
    flag 'kl_inside' marks the tokens whose KL is not capped.
    """
    lp = np.asarray(logp, dtype=np.float64)
    old = np.asarray(old_logp, dtype=np.float64)
    ref = np.asarray(ref_logp, dtype=np.float64)
    A = np.asarray(adv_tok, dtype=np.float64)
    rho = np.exp(lp - old)
    s1 = rho * A
    s2 = np.clip(rho, 1.0 - clip_eps, 1.0 + clip_eps) * A
    unclipped = s1 <= s2
    s = np.where(unclipped, s1, s2)
    d = ref - lp
    k3 = np.exp(d) - d - 1.0
    inside = ~(k3 > kl_clamp)
    kl = np.where(inside, k3, kl_clamp)
    return {"rho": rho, "s": s, "kl": kl, "ell": -s + beta * kl, "unclipped": unclipped, "kl_inside": inside}


def token_weights(mask, n_resp: int, L: int, agg_mode: int = 0, norm: float = 0.0) -> np.ndarray:
    """w_t so that loss = sum_t w_t l_t.

    agg_mode 0: mask_t / N_valid (token-mean; 0 when N_valid = 0).
    agg_mode 1: mask_t / (n_resp |o_i|), Eq. 1's per-response mean then mean
    over responses (a response with |o_i| = 0 contributes nothing).
    norm > 0 replaces N_valid (mode 0) or n_resp (mode 1): the count over the
    whole step's batch when this batch is one shard of it, since Eq. 1's
    expectation runs over every prompt of the step.
    """
    m = (np.asarray(mask) != 0).astype(np.float64)
    if agg_mode == 0:
        n = norm if norm > 0 else m.sum()
        return m / n if n > 0 else np.zeros_like(m)
    if agg_mode == 1:
        lens = m.reshape(n_resp, L).sum(axis=1)
        inv = np.where(lens > 0, 1.0 / np.maximum(lens, 1.0), 0.0) / (norm if norm > 0 else n_resp)
        return m * np.repeat(inv, L)
    raise ValueError(agg_mode)


def logp_coef(logp, old_logp, ref_logp, adv_tok, w, clip_eps: float, beta: float,
              kl_clamp: float = np.inf) -> np.ndarray:
    """g_t = dloss/dlogp_t = w_t (-A rho 1[unclipped] + beta (1 - exp(ref - logp)) 1[kl inside])."""
    tt = token_terms(logp, old_logp, ref_logp, adv_tok, clip_eps, beta, kl_clamp)
    lp = np.asarray(logp, dtype=np.float64)
    ref = np.asarray(ref_logp, dtype=np.float64)
    A = np.asarray(adv_tok, dtype=np.float64)
    dsurr = np.where(tt["unclipped"], A * tt["rho"], 0.0)
    dkl = np.where(tt["kl_inside"], 1.0 - np.exp(ref - lp), 0.0)
    return np.asarray(w, dtype=np.float64) * (-dsurr + beta * dkl)


def grpo_loss(logp, old_logp, ref_logp, adv, mask, n_resp: int, L: int,
              clip_eps: float, beta: float, agg_mode: int = 0, norm: float = 0.0, kl_clamp: float = np.inf):
    """Eq. 1 negated, from per-token log-probs. Returns (loss, g, per-token dict)."""
    A = token_advantages(adv, n_resp, L)
    w = token_weights(mask, n_resp, L, agg_mode, norm)
    tt = token_terms(logp, old_logp, ref_logp, A, clip_eps, beta, kl_clamp)
    m = np.asarray(mask) != 0
    loss = float(np.sum(w[m] * tt["ell"][m]))
    g = logp_coef(logp, old_logp, ref_logp, A, w, clip_eps, beta, kl_clamp)
    g[~m] = 0.0
    tt["w"] = w
    return loss, g, tt


# ---------------------------------------------------------------------------
# backward through the LM head
# ---------------------------------------------------------------------------


def loss_fwd_bwd(H, W, targets, mask, old_logp, ref_logp, adv, n_resp: int, L: int,
                 clip_eps: float, beta: float, agg_mode: int = 0, vocab_chunk: int = 8192,
                 norm: float = 0.0, kl_clamp: float = np.inf):
    """Full forward + backward: returns dict(loss, dH [T,Hd], dW [V,Hd], logp, lse, g)."""
    Hf = as_f64(H)
    Wf = as_f64(W)
    y = np.asarray(targets, dtype=np.int64)
    m = np.asarray(mask) != 0
    logp, lse = token_logprobs(Hf, Wf, y, m, vocab_chunk=vocab_chunk)
    loss, g, tt = grpo_loss(logp, old_logp, ref_logp, adv, m, n_resp, L, clip_eps, beta, agg_mode, norm,
                            kl_clamp)
    T, Hd = Hf.shape
    V = Wf.shape[0]
    dH = np.zeros((T, Hd))
    dW = np.zeros((V, Hd))
    idx = np.flatnonzero(m)
    if idx.size:
        Hv = Hf[idx]
        gv = g[idx]
        lv = lse[idx]
        yv = y[idx]
        dHv = np.zeros((idx.size, Hd))
        for v0 in range(0, V, vocab_chunk):
            v1 = min(V, v0 + vocab_chunk)
            Z = Hv @ Wf[v0:v1].T
            dZ = -gv[:, None] * np.exp(Z - lv[:, None])
            hit = np.flatnonzero((yv >= v0) & (yv < v1))
            dZ[hit, yv[hit] - v0] += gv[hit]
            dHv += dZ @ Wf[v0:v1]
            dW[v0:v1] = dZ.T @ Hv
        dH[idx] = dHv
    return {"loss": loss, "dH": dH, "dW": dW, "logp": logp, "lse": lse, "g": g, "terms": tt}


def dH_rows(H, W, targets, lse, g, rows, vocab_chunk: int = 8192) -> np.ndarray:
    """dH_t = g_t (W_{y_t} - sum_v p_{t,v} W_v) for the listed rows (any size)."""
    rows = np.asarray(rows, dtype=np.int64)
    Hf = as_f64(np.asarray(H)[rows])
    Wsrc = np.asarray(W)
    V = Wsrc.shape[0]
    y = np.asarray(targets, dtype=np.int64)[rows]
    l = np.asarray(lse, dtype=np.float64)[rows]
    gg = np.asarray(g, dtype=np.float64)[rows]
    acc = np.zeros((rows.size, Hf.shape[1]))
    for v0 in range(0, V, vocab_chunk):
        v1 = min(V, v0 + vocab_chunk)
        Wc = as_f64(Wsrc[v0:v1])
        P = np.exp(Hf @ Wc.T - l[:, None])
        acc += P @ Wc
    Wy = as_f64(Wsrc[y])
    return gg[:, None] * (Wy - acc)


def dW_rows(H, W, targets, mask, lse, g, vrows, row_chunk: int = 8192) -> np.ndarray:
    """dW_v = sum_t g_t (1[y_t = v] - p_{t,v}) H_t for the listed vocabulary rows (any size)."""
    vrows = np.asarray(vrows, dtype=np.int64)
    Wv = as_f64(np.asarray(W)[vrows])
    m = np.asarray(mask) != 0
    idx = np.flatnonzero(m)
    y = np.asarray(targets, dtype=np.int64)
    out = np.zeros((vrows.size, Wv.shape[1]))
    for r0 in range(0, idx.size, row_chunk):
        rows = idx[r0:r0 + row_chunk]
        Hr = as_f64(np.asarray(H)[rows])
        gr = np.asarray(g, dtype=np.float64)[rows]
        lr = np.asarray(lse, dtype=np.float64)[rows]
        P = np.exp(Hr @ Wv.T - lr[:, None])           # [rows, |vrows|]
        dZ = -gr[:, None] * P
        hit = y[rows][:, None] == vrows[None, :]
        dZ += hit * gr[:, None]
        out += dZ.T @ Hr
    return out


# ---------------------------------------------------------------------------
# the update that consumes dW: the actor's optimiser step
# ---------------------------------------------------------------------------


def adamw_step(theta, m, v, g, lr: float, beta1: float, beta2: float, eps: float,
               weight_decay: float, step: int):
    """One AdamW step (Adam with decoupled weight decay), float64.

    The paper fixes only the actor learning rate (1e-6, Section 4.1); the
    optimiser is read as AdamW:
        m <- beta1 m + (1 - beta1) g
        v <- beta2 v + (1 - beta2) g^2
        theta <- theta (1 - lr wd) - lr (m / (1 - beta1^t)) / (sqrt(v / (1 - beta2^t)) + eps)
    Returns (theta, m, v) as new arrays.
    """
    th = np.asarray(theta, dtype=np.float64)
    m1 = beta1 * np.asarray(m, dtype=np.float64) + (1.0 - beta1) * np.asarray(g, dtype=np.float64)
    v1 = beta2 * np.asarray(v, dtype=np.float64) + (1.0 - beta2) * np.asarray(g, dtype=np.float64) ** 2
    mhat = m1 / (1.0 - beta1 ** step)
    vhat = v1 / (1.0 - beta2 ** step)
    th1 = th * (1.0 - lr * weight_decay) - lr * mhat / (np.sqrt(vhat) + eps)
    return th1, m1, v1


# ---------------------------------------------------------------------------
# the rollout side: sampling o_{i,t} ~ pi_theta_old (Eq. 1's {o_i} ~ pi_old)
# ---------------------------------------------------------------------------


def gumbel_noise(seed: int, offset: int, rows, V: int, cols=None) -> np.ndarray:
    """G[t, v] = -log(-log U) with U the uniform of Philox4x32-10 word (v mod 4) at
    counter (v div 4, t, offset mod 2^32, offset div 2^32), key (seed mod 2^32, seed div 2^32).
    `rows` are token positions t; returns float64 [len(rows), V] (or [len(rows), len(cols)])."""
    from .philox import philox4x32_10, uniform_open
    t = np.asarray(rows, dtype=np.uint64)[:, None]
    v = np.arange(V, dtype=np.uint64) if cols is None else np.asarray(cols, dtype=np.uint64)
    words = philox4x32_10(v[None, :] >> np.uint64(2), t, offset & 0xFFFFFFFF, (offset >> 32) & 0xFFFFFFFF,
                          seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF)
    sel = (v & np.uint64(3))[None, :]
    w = np.where(sel == 0, words[0], np.where(sel == 1, words[1], np.where(sel == 2, words[2], words[3])))
    return -np.log(-np.log(uniform_open(w)))


def sample_tokens(H, W, mask, temperature: float, seed: int, offset: int, rows=None, vocab_chunk: int = 8192):
    """Gumbel-max sampling from softmax(H_t W^T / temperature) at the listed
    (or all unmasked) rows: y_t = argmax_v (z_{t,v} / temperature + G[t, v]),
    the lowest v on ties.  Returns (tokens int64 [-1 on masked], logp of the
    sampled token under softmax(z / temperature), gap between the best and
    second-best perturbed score) for every row (masked rows: -1, 0, inf)."""
    Hf = np.asarray(H)
    Wf = as_f64(W)
    T, V = Hf.shape[0], Wf.shape[0]
    m = np.asarray(mask) != 0
    idx = np.flatnonzero(m) if rows is None else np.asarray(rows, dtype=np.int64)
    tokens = np.full(T, -1, dtype=np.int64)
    logp = np.zeros(T)
    gap = np.full(T, np.inf)
    inv_t = 1.0 / temperature
    for r0 in range(0, idx.size, 256):
        rr = idx[r0:r0 + 256]
        rr = rr[m[rr]]
        if rr.size == 0:
            continue
        Hr = as_f64(Hf[rr])
        best = np.full(rr.size, -np.inf)
        second = np.full(rr.size, -np.inf)
        arg = np.zeros(rr.size, dtype=np.int64)
        zbest = np.zeros(rr.size)
        run_max = np.full(rr.size, -np.inf)
        run_sum = np.zeros(rr.size)
        for v0 in range(0, V, vocab_chunk):
            v1 = min(V, v0 + vocab_chunk)
            Z = (Hr @ Wf[v0:v1].T) * inv_t
            S = Z + gumbel_noise(seed, offset, rr, V, cols=np.arange(v0, v1))
            j = np.argmax(S, axis=1)
            sj = S[np.arange(rr.size), j]
            S2 = S.copy()
            S2[np.arange(rr.size), j] = -np.inf
            s2 = S2.max(axis=1)
            better = sj > best
            second = np.where(better, np.maximum(best, s2), np.maximum(second, sj))
            zbest = np.where(better, Z[np.arange(rr.size), j], zbest)
            arg = np.where(better, v0 + j, arg)
            best = np.where(better, sj, best)
            nm = np.maximum(run_max, Z.max(axis=1))
            run_sum = run_sum * np.exp(run_max - nm) + np.exp(Z - nm[:, None]).sum(axis=1)
            run_max = nm
        tokens[rr] = arg
        logp[rr] = zbest - (run_max + np.log(run_sum))
        gap[rr] = best - second
    return tokens, logp, gap


def nucleus(y, top_p: float):
    """Nucleus (top-p) set of softmax(y) for one row of tempered logits y: sort
    the tokens by probability, take the shortest prefix whose cumulative mass
    reaches top_p, and keep every token whose logit is at least that of the
    prefix's last token (so tokens tied with it are kept too).  top_p >= 1
    keeps the whole vocabulary.  Returns (bool mask, threshold logit, the
    set's probability mass)."""
    y = np.asarray(y, dtype=np.float64)
    if top_p >= 1.0:
        return np.ones(y.size, dtype=bool), -np.inf, 1.0
    mx = y.max()
    p = np.exp(y - (mx + np.log(np.exp(y - mx).sum())))
    order = np.argsort(-y, kind="stable")
    cum = np.cumsum(p[order])
    k = min(int(np.searchsorted(cum, top_p, side="left")), y.size - 1)
    thr = y[order[k]]
    keep = y >= thr
    return keep, thr, float(p[keep].sum())


def sample_tokens_top_p(H, W, mask, temperature: float, top_p: float, seed: int, offset: int, rows=None,
                        band_mass: float = 1e-5, band_logit: float = 1e-3):
    """Gumbel-max sampling restricted to the nucleus: y_t = argmax over v in
    nucleus(z_t / temperature, top_p) of (z_{t,v} / temperature + G[t, v]), the
    lowest v on ties, with the noise of gumbel_noise.  Returns, for every row
    (masked rows: -1, 0, inf, (inf, inf)): tokens, the log-prob of the sampled
    token under the untruncated softmax(z / temperature), the gap between the
    best and second-best perturbed score inside the nucleus, and the band of
    logits [lo, hi] whose membership could change if the cumulative masses
    moved by band_mass or the logits by band_logit (lower-precision
    arithmetic near the nucleus boundary)."""
    Hf = np.asarray(H)
    Wf = as_f64(W)
    T, V = Hf.shape[0], Wf.shape[0]
    m = np.asarray(mask) != 0
    idx = np.flatnonzero(m) if rows is None else np.asarray(rows, dtype=np.int64)
    idx = idx[m[idx]]
    tokens = np.full(T, -1, dtype=np.int64)
    logp = np.zeros(T)
    gap = np.full(T, np.inf)
    band = np.full((T, 2), np.inf)
    inv_t = 1.0 / temperature
    for r0 in range(0, idx.size, 32):
        rr = idx[r0:r0 + 32]
        Z = (as_f64(Hf[rr]) @ Wf.T) * inv_t
        G = gumbel_noise(seed, offset, rr, V)
        for i, t in enumerate(rr):
            y = Z[i]
            keep, _, _ = nucleus(y, top_p)
            S = np.where(keep, y + G[i], -np.inf)
            j = int(np.argmax(S))
            S[j] = -np.inf
            gap[t] = (y[j] + G[i, j]) - S.max() if keep.sum() > 1 else np.inf
            mx = y.max()
            lse = mx + np.log(np.exp(y - mx).sum())
            tokens[t] = j
            logp[t] = y[j] - lse
            if top_p >= 1.0:
                band[t] = (-np.inf, -np.inf)
            else:
                order = np.argsort(-y, kind="stable")
                cum = np.cumsum(np.exp(y[order] - lse))
                k_lo = min(int(np.searchsorted(cum, top_p - band_mass, side="left")), V - 1)
                k_hi = min(int(np.searchsorted(cum, top_p + band_mass, side="left")), V - 1)
                band[t] = (y[order[k_hi]] - band_logit, y[order[k_lo]] + band_logit)
    return tokens, logp, gap, band

