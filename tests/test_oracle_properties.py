"""Property pins of the float64 oracle over seeded random small shapes and values.

Each property follows from Eq. 1 / Eq. 2 of Section 3.3 or from the algebra of
the softmax, independently of how the oracle computes it:

* Eq. 2 is invariant to adding a constant to a group's rewards, and its
  advantages sum to zero within each group;
* the log-probs of all V possible targets of a row exponentiate to a
  distribution (sum 1), and match the brute-force loops;
* dH_t = g_t (W_{y_t} - sum_v p_{t,v} W_v): the gradient in closed form, a
  different route from the oracle's dZ @ W;
* relabelling the vocabulary (permuting W's rows and the targets alike)
  permutes dW's rows and leaves the loss and dH unchanged;
* with equal response lengths the token-mean and per-response-mean
  aggregations of Eq. 1 coincide.
"""
import numpy as np
import pytest

import oracle
from oracle import brute

EXAMPLES = 30


def _examples(draw_seed, /, **space):
    """EXAMPLES parameter sets drawn with a fixed seed: each key of `space` is an
    inclusive integer range (lo, hi) or a list of values to choose from."""
    rng = np.random.default_rng(draw_seed)
    out = []
    for _ in range(EXAMPLES):
        ex = {}
        for k, v in space.items():
            ex[k] = int(rng.integers(v[0], v[1] + 1)) if isinstance(v, tuple) else v[int(rng.integers(len(v)))]
        out.append(ex)
    return out


def _cases(draw_seed, /, **space):
    exs = _examples(draw_seed, **space)
    names = list(space)
    return pytest.mark.parametrize(",".join(names), [tuple(e[n] for n in names) for e in exs])


def _case(seed, n_groups, G, L, Hd, V, ragged=True):
    rng = np.random.default_rng(seed)
    n_resp = n_groups * G
    T = n_resp * L
    H = rng.normal(0, 1, (T, Hd))
    W = rng.normal(0, 0.7, (V, Hd))
    y = rng.integers(0, V, T)
    lens = rng.integers(1, L + 1, n_resp) if ragged else np.full(n_resp, L)
    m = (np.arange(L)[None, :] < lens[:, None]).astype(np.uint8).reshape(-1)
    r = rng.choice([0.0, 0.5, 1.0], n_resp)
    return rng, H, W, y, m, r, n_resp


@_cases(101, seed=(0, 10**6), n_groups=(1, 5), G=(2, 16), shift=[-3.0, -0.5, 0.25, 2.0])
def test_advantages_shift_invariant_and_zero_mean(seed, n_groups, G, shift):
    rng = np.random.default_rng(seed)
    r = rng.choice([0.0, 0.5, 1.0], n_groups * G)  # dyadic: the shifted sums stay exact
    a = oracle.group_advantages(r, G).astype(np.float64)
    b = oracle.group_advantages(r + shift, G).astype(np.float64)
    np.testing.assert_allclose(a, b, rtol=0, atol=2e-7)
    assert np.all(np.abs(a.reshape(n_groups, G).sum(1)) <= 1e-5 * G)


@_cases(102, seed=(0, 10**6), T=(1, 6), Hd=(1, 6), V=(2, 12))
def test_logprobs_form_a_distribution_and_match_brute_force(seed, T, Hd, V):
    rng = np.random.default_rng(seed)
    H, W = rng.normal(0, 1.5, (T, Hd)), rng.normal(0, 1.5, (V, Hd))
    m = np.ones(T, np.uint8)
    allv = np.stack([oracle.token_logprobs(H, W, np.full(T, v), m)[0] for v in range(V)], 1)
    np.testing.assert_allclose(np.exp(allv).sum(1), 1.0, rtol=1e-12)
    assert np.all(allv <= 0)
    y = rng.integers(0, V, T)
    got = oracle.token_logprobs(H, W, y, m)[0]
    np.testing.assert_allclose(got, brute.logprobs(H.tolist(), W.tolist(), y.tolist(), m.tolist()),
                               rtol=1e-12, atol=1e-12)


@_cases(103, seed=(0, 10**6), n_groups=(1, 3), G=(2, 4), L=(1, 5), Hd=(1, 6), V=(2, 10))
def test_dH_closed_form_and_vocabulary_relabelling(seed, n_groups, G, L, Hd, V):
    rng, H, W, y, m, r, n_resp = _case(seed, n_groups, G, L, Hd, V)
    logp, _ = oracle.token_logprobs(H, W, y, m)
    old = logp - rng.normal(0, 0.3, logp.size)
    ref = logp + rng.normal(0, 0.3, logp.size)
    adv = oracle.group_advantages(r, G)
    out = oracle.loss_fwd_bwd(H, W, y, m, old, ref, adv, n_resp, L, 0.2, 0.04, 0, vocab_chunk=3)
    # closed form of dH
    Z = H @ W.T
    P = np.exp(Z - out["lse"][:, None])
    want = out["g"][:, None] * (W[y] - P @ W)
    want[m == 0] = 0.0
    np.testing.assert_allclose(out["dH"], want, rtol=1e-9, atol=1e-13)
    # relabel the vocabulary
    perm = rng.permutation(V)
    inv = np.argsort(perm)
    out2 = oracle.loss_fwd_bwd(H, W[perm], inv[y], m, old, ref, adv, n_resp, L, 0.2, 0.04, 0, vocab_chunk=4)
    assert out2["loss"] == pytest.approx(out["loss"], rel=1e-12, abs=1e-15)
    np.testing.assert_allclose(out2["dH"], out["dH"], rtol=1e-10, atol=1e-14)
    np.testing.assert_allclose(out2["dW"], out["dW"][perm], rtol=1e-10, atol=1e-14)


@_cases(104, seed=(0, 10**6), n_groups=(1, 3), G=(2, 4), L=(1, 5))
def test_aggregations_agree_for_equal_lengths(seed, n_groups, G, L):
    rng, H, W, y, m, r, n_resp = _case(seed, n_groups, G, L, 3, 5, ragged=False)
    logp, _ = oracle.token_logprobs(H, W, y, m)
    old = logp - rng.normal(0, 0.3, logp.size)
    ref = logp + rng.normal(0, 0.3, logp.size)
    adv = oracle.group_advantages(r, G)
    a = oracle.grpo_loss(logp, old, ref, adv, m, n_resp, L, 0.2, 0.04, 0)
    b = oracle.grpo_loss(logp, old, ref, adv, m, n_resp, L, 0.2, 0.04, 1)
    assert a[0] == pytest.approx(b[0], rel=1e-12, abs=1e-15)
    np.testing.assert_allclose(a[1], b[1], rtol=1e-12, atol=1e-15)
