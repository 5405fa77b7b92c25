"""Pins of the float64 oracle against facts that do not come from the oracle itself.

Each pin is a closed form, a brute-force loop, a library routine, an invariant
or a finite-difference check of Eq. 1 / Eq. 2 (Section 3.3).  The last block
plants plausible mistakes into a copy of the oracle and checks that a pin
catches each one.
"""
import json
import math
import os
import statistics
import struct

import numpy as np
import pytest
import scipy.special

import oracle
from oracle import brute
from oracle import grpo_oracle as go

HERE = os.path.dirname(os.path.abspath(__file__))


def _rand_case(seed, T_resp=3, G=2, L=4, Hd=5, V=7, scale=0.7, ragged=True):
    """A tiny float64 case with ragged prefix masks and non-degenerate advantages."""
    rng = np.random.default_rng(seed)
    n_resp = T_resp * G if T_resp else G
    T = n_resp * L
    H = rng.normal(0, 1, (T, Hd))
    W = rng.normal(0, scale, (V, Hd))
    y = rng.integers(0, V, T)
    lens = rng.integers(1, L + 1, n_resp) if ragged else np.full(n_resp, L)
    mask = (np.arange(L)[None, :] < lens[:, None]).astype(np.uint8).reshape(-1)
    r = np.tile(np.array([0.0, 1.0] * (G // 2) + [0.5] * (G % 2)), n_resp // G)
    rng.shuffle(r)
    return dict(H=H, W=W, y=y, mask=mask, rewards=r, n_resp=n_resp, L=L, G=G, rng=rng)


def _old_ref(logp, rng, spread=(-0.6, -0.05, 0.07, 0.5)):
    """old/ref log-probs at fixed offsets from logp, so rho sits well away from 1 +- eps."""
    off_old = rng.choice(spread, size=logp.size)
    off_ref = rng.normal(0, 0.3, size=logp.size)
    return logp - off_old, logp + off_ref


# ---------------------------------------------------------------------------
# Eq. 2
# ---------------------------------------------------------------------------

def test_advantage_closed_forms():
    fx = json.load(open(os.path.join(HERE, "golden", "advantage_closed_forms.json")))
    for c in fx["cases"]:
        got = oracle.group_advantages(np.array(c["rewards"], np.float32), c["G"], fx["eps"])
        np.testing.assert_allclose(got, np.array(c["adv"], np.float32), rtol=0, atol=2e-7)
        assert statistics.stdev(c["rewards"]) == pytest.approx(c["std"], abs=1e-15)
        assert statistics.mean(c["rewards"]) == pytest.approx(c["mean"], abs=1e-15)


def test_advantages_zero_mean_and_library_std():
    rng = np.random.default_rng(3)
    for G in (2, 3, 4, 8, 16, 64):
        r = rng.random(G * 5).astype(np.float32)
        a = oracle.group_advantages(r, G, eps=0.0).astype(np.float64).reshape(-1, G)
        assert np.abs(a.sum(axis=1)).max() < 1e-5
        # with eps = 0 every group has sample std exactly 1 after normalisation
        for row in a:
            assert statistics.stdev(row.tolist()) == pytest.approx(1.0, abs=1e-6)
        # brute-force loop
        bf = np.array(brute.advantages(r.tolist(), G), np.float32)
        np.testing.assert_allclose(oracle.group_advantages(r, G), bf, rtol=0, atol=1e-6)


def test_advantages_all_equal_group_is_zero_and_bad_group_rejected():
    r = np.array([0.5] * 8 + [1, 0, 0, 0, 0, 0, 0, 0], np.float32)
    a = oracle.group_advantages(r, 8)
    assert np.all(a[:8] == 0.0)
    with pytest.raises(ValueError):
        oracle.group_advantages(r, 1)
    with pytest.raises(ValueError):
        oracle.group_advantages(r[:7], 4)


# ---------------------------------------------------------------------------
# pi_theta(o_t): log-softmax at the sampled token
# ---------------------------------------------------------------------------

def test_uniform_logits_give_minus_log_V():
    rng = np.random.default_rng(0)
    for V in (7, 4096, 10001):
        T, Hd = 9, 16
        H = rng.normal(size=(T, Hd))
        y = rng.integers(0, V, T)
        mask = np.ones(T, np.uint8)
        logp, lse = oracle.token_logprobs(H, np.zeros((V, Hd)), y, mask, vocab_chunk=1000)
        assert np.all(logp == -np.log(V)) or np.abs(logp + math.log(V)).max() < 1e-12
        logp0, _ = oracle.token_logprobs(np.zeros((T, Hd)), rng.normal(size=(V, Hd)), y, mask)
        assert np.abs(logp0 + math.log(V)).max() < 1e-12


def test_logprobs_match_bruteforce_and_scipy():
    c = _rand_case(1, T_resp=2, G=2, L=5, Hd=6, V=11, scale=1.5)
    logp, lse = oracle.token_logprobs(c["H"], c["W"], c["y"], c["mask"], vocab_chunk=4)
    bf = brute.logprobs(c["H"].tolist(), c["W"].tolist(), c["y"].tolist(), c["mask"].tolist())
    np.testing.assert_allclose(logp, bf, rtol=0, atol=1e-12)
    Z = c["H"] @ c["W"].T
    ls = scipy.special.log_softmax(Z, axis=1)[np.arange(len(c["y"])), c["y"]]
    m = c["mask"] != 0
    np.testing.assert_allclose(logp[m], ls[m], rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse[m], scipy.special.logsumexp(Z, axis=1)[m], rtol=0, atol=1e-12)
    assert np.all(logp[~m] == 0) and np.all(lse[~m] == 0)


def test_target_logits_match_explicit_sums_and_logp_plus_lse():
    """z_{t,y_t} against dot products written out in pure Python (bf16 inputs
    widened bit by bit), and logp_t = z_{t,y_t} - LSE_t against brute force."""
    rng = np.random.default_rng(17)
    T, Hd, V = 9, 7, 13
    Hb = rng.integers(0, 1 << 16, (T, Hd), dtype=np.uint16) & np.uint16(0xBFFF)   # finite bf16 bit patterns
    Wb = rng.integers(0, 1 << 16, (V, Hd), dtype=np.uint16) & np.uint16(0xBFFF)
    y = rng.integers(0, V, T)
    rows = np.array([0, 3, 4, 8])

    def bits(b):
        return struct.unpack("<f", struct.pack("<I", int(b) << 16))[0]
    want = [math.fsum(bits(Hb[t, k]) * bits(Wb[y[t], k]) for k in range(Hd)) for t in rows]
    np.testing.assert_allclose(oracle.target_logits(Hb, Wb, y, rows), want, rtol=1e-13, atol=0)
    c = _rand_case(3, T_resp=2, G=2, L=4, Hd=5, V=9, scale=1.2)
    m = c["mask"] != 0
    logp, lse = oracle.token_logprobs(c["H"], c["W"], c["y"], c["mask"])
    idx = np.flatnonzero(m)
    bf = np.array(brute.logprobs(c["H"].tolist(), c["W"].tolist(), c["y"].tolist(), c["mask"].tolist()))
    np.testing.assert_allclose(oracle.target_logits(c["H"], c["W"], c["y"], idx) - lse[idx], bf[idx],
                               rtol=0, atol=1e-12)


def test_logprobs_chunking_invariant_and_large_logits():
    rng = np.random.default_rng(5)
    H = rng.normal(size=(20, 8))
    W = rng.normal(0, 30.0, size=(50, 8))   # logits in the hundreds: needs the max shift
    y = rng.integers(0, 50, 20)
    mask = np.ones(20, np.uint8)
    a, _ = oracle.token_logprobs(H, W, y, mask, vocab_chunk=3, row_chunk=7)
    b, _ = oracle.token_logprobs(H, W, y, mask, vocab_chunk=50)
    np.testing.assert_allclose(a, b, rtol=0, atol=1e-9)
    ls = scipy.special.log_softmax(H @ W.T, axis=1)[np.arange(20), y]
    np.testing.assert_allclose(a, ls, rtol=0, atol=1e-9)


def test_bf16_widening_is_exact():
    bits = np.array([0x3F80, 0xBF80, 0x0000, 0x4049, 0x7F7F, 0x0001], np.uint16)
    want = np.array([1.0, -1.0, 0.0, 3.140625, 3.3895313892515355e38, 9.183549615799121e-41])
    np.testing.assert_array_equal(oracle.widen_bf16(bits), want)


# ---------------------------------------------------------------------------
# Eq. 1: ratio, clip, KL, aggregation
# ---------------------------------------------------------------------------

def test_ratio_one_and_kl_zero_closed_forms():
    c = _rand_case(2, T_resp=2, G=4, L=6)
    logp, _ = oracle.token_logprobs(c["H"], c["W"], c["y"], c["mask"])
    adv = oracle.group_advantages(c["rewards"], c["G"])
    A = oracle.token_advantages(adv, c["n_resp"], c["L"])
    m = c["mask"] != 0
    ref = logp + c["rng"].normal(0, 0.3, logp.size)
    for agg in (0, 1):
        w = oracle.token_weights(c["mask"], c["n_resp"], c["L"], agg)
        # old = policy: rho = 1 -> loss = -sum w A + beta sum w KL
        loss, _, tt = oracle.grpo_loss(logp, logp, ref, adv, c["mask"], c["n_resp"], c["L"], 0.2, 0.04, agg)
        assert np.all(tt["rho"][m] == 1.0)
        d = ref - logp
        kl = np.exp(d) - d - 1
        assert loss == pytest.approx(float(np.sum(w[m] * (-A[m] + 0.04 * kl[m]))), abs=1e-14)
        # ref = policy too: KL = 0 -> loss = -sum w A
        loss2, _, tt2 = oracle.grpo_loss(logp, logp, logp, adv, c["mask"], c["n_resp"], c["L"], 0.2, 0.04, agg)
        assert np.all(tt2["kl"][m] == 0.0)
        assert loss2 == pytest.approx(-float(np.sum(w[m] * A[m])), abs=1e-14)


def test_token_mean_of_zero_mean_advantages_is_zero_for_equal_lengths():
    c = _rand_case(4, T_resp=3, G=4, L=5, ragged=False)
    logp, _ = oracle.token_logprobs(c["H"], c["W"], c["y"], c["mask"])
    adv = oracle.group_advantages(c["rewards"], c["G"])
    for agg in (0, 1):
        loss, _, _ = oracle.grpo_loss(logp, logp, logp, adv, c["mask"], c["n_resp"], c["L"], 0.2, 0.04, agg)
        assert abs(loss) < 1e-7  # float32 advantages sum to 0 up to rounding
    w0 = oracle.token_weights(c["mask"], c["n_resp"], c["L"], 0)
    w1 = oracle.token_weights(c["mask"], c["n_resp"], c["L"], 1)
    np.testing.assert_allclose(w0, w1, rtol=1e-15)


def test_kl_nonnegative_and_zero_only_at_equality():
    rng = np.random.default_rng(7)
    lp = rng.normal(-8, 2, 10000)
    ref = lp + rng.normal(0, 1, lp.size)
    tt = oracle.token_terms(lp, lp, ref, np.ones_like(lp), 0.2, 0.04)
    assert np.all(tt["kl"] >= 0)
    assert np.all(tt["kl"][np.abs(ref - lp) > 1e-3] > 0)
    # second-order: KL ~ d^2/2 for small d = ref - logp
    d = np.array([1e-3, -2e-3, 5e-4])
    tt = oracle.token_terms(np.zeros(3), np.zeros(3), d, np.ones(3), 0.2, 0.04)
    np.testing.assert_allclose(tt["kl"], d ** 2 / 2 + d ** 3 / 6, rtol=1e-3)


def test_loss_matches_bruteforce_both_aggregations():
    for seed in (11, 12, 13):
        c = _rand_case(seed, T_resp=3, G=4, L=5)
        logp, _ = oracle.token_logprobs(c["H"], c["W"], c["y"], c["mask"])
        old, ref = _old_ref(logp, c["rng"])
        adv = oracle.group_advantages(c["rewards"], c["G"])
        for agg in (0, 1):
            loss, _, _ = oracle.grpo_loss(logp, old, ref, adv, c["mask"], c["n_resp"], c["L"], 0.2, 0.04, agg)
            bl = brute.loss(logp.tolist(), old.tolist(), ref.tolist(), adv.astype(float).tolist(),
                            c["mask"].tolist(), c["n_resp"], c["L"], 0.2, 0.04, agg)
            assert loss == pytest.approx(bl, rel=1e-12, abs=1e-15)


def test_clip_zeroes_surrogate_gradient():
    lp = np.zeros(4)
    old = np.array([-0.5, 0.5, -0.5, 0.5])          # rho = e^0.5, e^-0.5, e^0.5, e^-0.5
    A = np.array([1.0, -1.0, -1.0, 1.0])
    g = oracle.logp_coef(lp, old, lp, A, np.ones(4), 0.2, 0.0)
    # A > 0, rho > 1 + eps and A < 0, rho < 1 - eps: clipped, no gradient
    assert g[0] == 0.0 and g[1] == 0.0
    # the other two stay on the unclipped branch: g = -A rho
    np.testing.assert_allclose(g[2:], [math.exp(0.5), -math.exp(-0.5)], rtol=1e-15)


def test_textbook_policy_gradient_special_case():
    c = _rand_case(21, T_resp=2, G=4, L=4)
    logp, _ = oracle.token_logprobs(c["H"], c["W"], c["y"], c["mask"])
    old, ref = _old_ref(logp, c["rng"])
    adv = oracle.group_advantages(c["rewards"], c["G"])
    A = oracle.token_advantages(adv, c["n_resp"], c["L"])
    w = oracle.token_weights(c["mask"], c["n_resp"], c["L"], 0)
    g = oracle.logp_coef(logp, old, ref, A, w, np.inf, 0.0)
    np.testing.assert_allclose(g, -w * A * np.exp(logp - old), rtol=1e-15)


# ---------------------------------------------------------------------------
# gradients
# ---------------------------------------------------------------------------

def _loss_of(H, W, c, old, ref, adv, agg, clip=0.2, beta=0.04):
    logp = brute.logprobs(H.tolist(), W.tolist(), c["y"].tolist(), c["mask"].tolist())
    return brute.loss(logp, old.tolist(), ref.tolist(), adv.astype(float).tolist(),
                      c["mask"].tolist(), c["n_resp"], c["L"], clip, beta, agg)


@pytest.mark.parametrize("agg", [0, 1])
def test_gradient_matches_central_differences(agg):
    c = _rand_case(31, T_resp=2, G=2, L=3, Hd=4, V=6, scale=0.8)
    logp, _ = oracle.token_logprobs(c["H"], c["W"], c["y"], c["mask"])
    old, ref = _old_ref(logp, c["rng"])
    adv = oracle.group_advantages(c["rewards"], c["G"])
    out = oracle.loss_fwd_bwd(c["H"], c["W"], c["y"], c["mask"], old, ref, adv, c["n_resp"], c["L"],
                              0.2, 0.04, agg, vocab_chunk=4)
    h = 1e-6
    for name, X, dX in (("H", c["H"], out["dH"]), ("W", c["W"], out["dW"])):
        fd = np.zeros_like(X)
        for i in range(X.shape[0]):
            for j in range(X.shape[1]):
                Xp = X.copy(); Xp[i, j] += h
                Xm = X.copy(); Xm[i, j] -= h
                args_p = (Xp, c["W"]) if name == "H" else (c["H"], Xp)
                args_m = (Xm, c["W"]) if name == "H" else (c["H"], Xm)
                fd[i, j] = (_loss_of(*args_p, c, old, ref, adv, agg) - _loss_of(*args_m, c, old, ref, adv, agg)) / (2 * h)
        np.testing.assert_allclose(dX, fd, rtol=1e-5, atol=1e-9, err_msg=name)
    assert np.all(out["dH"][c["mask"] == 0] == 0.0)


def _clamp_case(seed=33, kl_clamp=0.15):
    """A tiny case whose per-token k3 values lie on both sides of kl_clamp, each
    at least 0.02 away from it (finite differences stay on one side)."""
    c = _rand_case(seed, T_resp=2, G=2, L=3, Hd=4, V=6, scale=0.8)
    logp, _ = oracle.token_logprobs(c["H"], c["W"], c["y"], c["mask"])
    old, _ = _old_ref(logp, c["rng"])
    d = np.tile([-1.2, -0.2, 0.9, 0.1, 1.6, -0.5], logp.size // 6 + 1)[:logp.size]
    ref = logp + d
    k3 = np.exp(d) - d - 1.0
    m = c["mask"] != 0
    assert np.any(k3[m] > kl_clamp + 0.02) and np.any(k3[m] < kl_clamp - 0.02)
    assert np.all(np.abs(k3 - kl_clamp) > 0.02)
    return c, old, ref


def test_clamped_kl_gradient_matches_central_differences():
    kappa, beta = 0.15, 0.3
    c, old, ref = _clamp_case(kl_clamp=kappa)
    adv = oracle.group_advantages(c["rewards"], c["G"])
    out = oracle.loss_fwd_bwd(c["H"], c["W"], c["y"], c["mask"], old, ref, adv, c["n_resp"], c["L"],
                              0.2, beta, 0, vocab_chunk=4, kl_clamp=kappa)
    logp = oracle.token_logprobs(c["H"], c["W"], c["y"], c["mask"])[0]
    bl = brute.loss(logp.tolist(), old.tolist(), ref.tolist(), adv.astype(float).tolist(), c["mask"].tolist(),
                    c["n_resp"], c["L"], 0.2, beta, 0, kl_clamp=kappa)
    assert out["loss"] == pytest.approx(bl, rel=1e-12, abs=1e-15)
    h = 1e-6

    def f(H, W):
        lp = brute.logprobs(H.tolist(), W.tolist(), c["y"].tolist(), c["mask"].tolist())
        return brute.loss(lp, old.tolist(), ref.tolist(), adv.astype(float).tolist(), c["mask"].tolist(),
                          c["n_resp"], c["L"], 0.2, beta, 0, kl_clamp=kappa)
    for name, X, dX in (("H", c["H"], out["dH"]), ("W", c["W"], out["dW"])):
        fd = np.zeros_like(X)
        for i in range(X.shape[0]):
            for j in range(X.shape[1]):
                Xp = X.copy(); Xp[i, j] += h
                Xm = X.copy(); Xm[i, j] -= h
                fp = f(Xp, c["W"]) if name == "H" else f(c["H"], Xp)
                fm = f(Xm, c["W"]) if name == "H" else f(c["H"], Xm)
                fd[i, j] = (fp - fm) / (2 * h)
        np.testing.assert_allclose(dX, fd, rtol=1e-5, atol=1e-9, err_msg=name)


def test_kl_clamp_special_cases():
    """A cap of 0 removes the KL term (k3 >= 0), so the result is that of beta = 0;
    a cap above every k3 is the plain estimator, bit for bit."""
    c, old, ref = _clamp_case()
    adv = oracle.group_advantages(c["rewards"], c["G"])
    args = (c["H"], c["W"], c["y"], c["mask"], old, ref, adv, c["n_resp"], c["L"], 0.2)
    zero = oracle.loss_fwd_bwd(*args, 0.3, 0, vocab_chunk=4, kl_clamp=0.0)
    nokl = oracle.loss_fwd_bwd(*args, 0.0, 0, vocab_chunk=4)
    assert zero["loss"] == pytest.approx(nokl["loss"], rel=1e-12, abs=1e-15)
    np.testing.assert_allclose(zero["dH"], nokl["dH"], rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(zero["dW"], nokl["dW"], rtol=1e-12, atol=1e-15)
    big = oracle.loss_fwd_bwd(*args, 0.3, 0, vocab_chunk=4, kl_clamp=1e30)
    plain = oracle.loss_fwd_bwd(*args, 0.3, 0, vocab_chunk=4)
    assert big["loss"] == plain["loss"]
    assert np.array_equal(big["dH"], plain["dH"]) and np.array_equal(big["dW"], plain["dW"])
    # capped tokens carry exactly the cap as their KL value
    tt = plain["terms"]
    kt = oracle.token_terms(plain["logp"], old, ref, np.zeros_like(old), 0.2, 0.3, 0.15)
    capped = ~kt["kl_inside"]
    assert capped.any() and np.all(kt["kl"][capped] == 0.15)
    assert np.array_equal(kt["kl"][~capped], tt["kl"][~capped])


def test_dW_column_sums_vanish_and_sampled_rows_match():
    c = _rand_case(41, T_resp=3, G=4, L=6, Hd=8, V=23)
    logp, _ = oracle.token_logprobs(c["H"], c["W"], c["y"], c["mask"])
    old, ref = _old_ref(logp, c["rng"])
    adv = oracle.group_advantages(c["rewards"], c["G"])
    out = oracle.loss_fwd_bwd(c["H"], c["W"], c["y"], c["mask"], old, ref, adv, c["n_resp"], c["L"],
                              0.2, 0.04, 0, vocab_chunk=5)
    # sum_v dZ_{t,v} = 0 for every t, hence sum_v dW[v, :] = 0
    assert np.abs(out["dW"].sum(axis=0)).max() < 1e-13
    rows = np.flatnonzero(c["mask"])[::3]
    np.testing.assert_allclose(oracle.dH_rows(c["H"], c["W"], c["y"], out["lse"], out["g"], rows, vocab_chunk=4),
                               out["dH"][rows], rtol=1e-10, atol=1e-14)
    vrows = np.array([0, 5, 22, int(c["y"][np.flatnonzero(c["mask"])[0]])])
    np.testing.assert_allclose(oracle.dW_rows(c["H"], c["W"], c["y"], c["mask"], out["lse"], out["g"], vrows, row_chunk=5),
                               out["dW"][vrows], rtol=1e-10, atol=1e-14)
    # dH_t = g_t (W_{y_t} - E_p[W])
    t = rows[0]
    z = c["W"] @ c["H"][t]
    p = np.exp(z - scipy.special.logsumexp(z))
    np.testing.assert_allclose(out["dH"][t], out["g"][t] * (c["W"][c["y"][t]] - p @ c["W"]), rtol=1e-10)


def test_all_masked_batch_is_zero():
    c = _rand_case(51, T_resp=1, G=2, L=3)
    mask = np.zeros_like(c["mask"])
    zeros = np.zeros(mask.size)
    adv = oracle.group_advantages(c["rewards"], c["G"])
    out = oracle.loss_fwd_bwd(c["H"], c["W"], c["y"], mask, zeros, zeros, adv, c["n_resp"], c["L"], 0.2, 0.04)
    assert out["loss"] == 0.0 and not out["dH"].any() and not out["dW"].any()


# ---------------------------------------------------------------------------
# the optimiser step that consumes dW
# ---------------------------------------------------------------------------

def test_adamw_first_step_closed_form():
    g = np.array([3.0, -2e-3, 0.5, 0.0])
    th = np.array([1.0, -1.0, 0.25, 2.0])
    lr, wd, eps = 1e-3, 0.01, 1e-8
    t1, m1, v1 = oracle.adamw_step(th, np.zeros(4), np.zeros(4), g, lr, 0.9, 0.999, eps, wd, 1)
    # step 1 from zero moments: m_hat = g, v_hat = g^2
    np.testing.assert_allclose(m1, 0.1 * g, rtol=1e-15)
    np.testing.assert_allclose(v1, 0.001 * g * g, rtol=1e-15)
    np.testing.assert_allclose(t1, th * (1 - lr * wd) - lr * g / (np.abs(g) + eps), rtol=1e-12)


def test_adamw_matches_torch_optimizer():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(9)
    th0 = rng.normal(size=(5, 7))
    grads = [rng.normal(size=(5, 7)) * s for s in (1.0, 0.3, 2.0)]
    p = torch.nn.Parameter(torch.from_numpy(th0.copy()))
    opt = torch.optim.AdamW([p], lr=1e-3, betas=(0.9, 0.95), eps=1e-8, weight_decay=0.1)
    th, m, v = th0, np.zeros_like(th0), np.zeros_like(th0)
    for t, g in enumerate(grads, start=1):
        p.grad = torch.from_numpy(g.copy())
        opt.step()
        th, m, v = oracle.adamw_step(th, m, v, g, 1e-3, 0.9, 0.95, 1e-8, 0.1, t)
    np.testing.assert_allclose(th, p.detach().numpy(), rtol=0, atol=1e-13)
    st = opt.state[p]
    np.testing.assert_allclose(m, st["exp_avg"].numpy(), rtol=1e-13)
    np.testing.assert_allclose(v, st["exp_avg_sq"].numpy(), rtol=1e-13)


# ---------------------------------------------------------------------------
# sampling: Philox4x32-10 and the Gumbel-max draw
# ---------------------------------------------------------------------------

def test_philox_known_answer_vectors():
    """The known-answer vectors published with the generator's reference implementation."""
    from oracle import philox
    cases = [((0, 0, 0, 0), (0, 0), (0x6627E8D5, 0xE169C58D, 0xBC57AC4C, 0x9B00DBD8)),
             ((0xFFFFFFFF,) * 4, (0xFFFFFFFF,) * 2, (0x408F276D, 0x41C83B0E, 0xA20BC7C6, 0x6D5451FD)),
             ((0x243F6A88, 0x85A308D3, 0x13198A2E, 0x03707344), (0xA4093822, 0x299F31D0),
              (0xD16CFE09, 0x94FDCCEB, 0x5001E420, 0x24126EA1))]
    for ctr, key, want in cases:
        assert [int(x) for x in philox.philox4x32_10(*ctr, *key)] == list(want)
    u = philox.uniform_open(np.array([0, 511, 512, 0xFFFFFFFF], dtype=np.uint64))
    np.testing.assert_array_equal(u, [0.5 / 2 ** 23, 0.5 / 2 ** 23, 1.5 / 2 ** 23, 1 - 0.5 / 2 ** 23])


def test_gumbel_max_samples_follow_the_softmax():
    """Many rows with the same logits: the sampled tokens' frequencies follow softmax(z / tau)."""
    from scipy.stats import chisquare
    V, T, Hd = 6, 30000, 3
    W = np.array([[1.0, 0, 0], [0.5, 0, 0], [0, 1, 0], [0, 0, 1], [-1.0, 0, 0], [0.2, 0.2, 0.2]])
    H = np.tile(np.array([[0.9, -0.4, 0.3]]), (T, 1))
    z = W @ H[0]
    for tau in (1.0, 0.5, 2.0):
        tok, logp, _ = oracle.sample_tokens(H, W, np.ones(T, np.uint8), tau, seed=1234, offset=7)
        p = scipy.special.softmax(z / tau)
        counts = np.bincount(tok, minlength=V)
        assert chisquare(counts, p * T).pvalue > 1e-4
        np.testing.assert_allclose(logp, np.log(p)[tok], rtol=0, atol=1e-12)
    tok, _, _ = oracle.sample_tokens(H[:50], W, np.ones(50, np.uint8), 1e-3, seed=5, offset=0)
    assert np.all(tok == np.argmax(z))  # tau -> 0: greedy


def test_sampling_counter_layout():
    """Rows, offsets and seeds index disjoint noise; word v mod 4 of counter v div 4."""
    from oracle import philox
    g = oracle.gumbel_noise(99, 5, [3, 4], 9)
    w = philox.philox4x32_10(2, 3, 5, 0, 99, 0)
    assert g[0, 9 - 1] == -np.log(-np.log(philox.uniform_open(w[0])))   # v = 8 -> counter 2, word 0
    assert not np.array_equal(g[0], g[1])
    assert not np.array_equal(g, oracle.gumbel_noise(99, 6, [3, 4], 9))
    assert not np.array_equal(g, oracle.gumbel_noise(98, 5, [3, 4], 9))


def _nucleus_by_threshold_search(y, top_p):
    """The nucleus as the highest logit threshold whose upper set reaches
    top_p, searched over the row's distinct logit values with explicit sums."""
    p = [math.exp(v) for v in y]
    total = math.fsum(p)
    for thr in sorted(set(y), reverse=True):
        if math.fsum(pv for pv, v in zip(p, y) if v >= thr) / total >= top_p:
            return np.array([v >= thr for v in y])
    return np.ones(len(y), dtype=bool)


def test_nucleus_matches_threshold_search():
    """Random rows with many ties (logits on a half-integer grid): the nucleus
    equals the threshold search, keeps whole tie groups, and drops below top_p
    without its lowest tie group."""
    rng = np.random.default_rng(31)
    for _ in range(400):
        V = int(rng.integers(1, 13))
        y = (rng.integers(-4, 5, V) / 2.0).tolist()
        top_p = float(rng.choice([rng.uniform(0.01, 0.99), 0.5, 0.9, 1.0]))
        keep, thr, mass = oracle.nucleus(np.array(y), top_p)
        want = _nucleus_by_threshold_search(y, top_p)
        np.testing.assert_array_equal(keep, want)
        if top_p < 1.0:
            p = scipy.special.softmax(np.array(y))
            assert mass >= top_p - 1e-12
            assert p[np.array(y) > thr].sum() < top_p


def test_top_p_draws_follow_the_truncated_softmax():
    """Many rows with the same logits: inside the nucleus the sampled tokens'
    frequencies follow the softmax renormalised on it, outside they never
    occur; top_p = 1 is the plain sampler, a tiny top_p the greedy one."""
    from scipy.stats import chisquare
    V, T = 6, 30000
    W = np.array([[1.0, 0, 0], [0.5, 0, 0], [0, 1, 0], [0, 0, 1], [-1.0, 0, 0], [0.2, 0.2, 0.2]])
    H = np.tile(np.array([[0.9, -0.4, 0.3]]), (T, 1))
    z = W @ H[0]
    ones = np.ones(T, np.uint8)
    for tau, top_p in ((1.0, 0.6), (0.5, 0.8), (2.0, 0.5)):
        p = scipy.special.softmax(z / tau)
        keep = oracle.nucleus(z / tau, top_p)[0]
        assert 1 < keep.sum() < V
        tok, logp, _, _ = oracle.sample_tokens_top_p(H, W, ones, tau, top_p, seed=1234, offset=7)
        counts = np.bincount(tok, minlength=V)
        assert counts[~keep].sum() == 0
        q = p[keep] / p[keep].sum()
        assert chisquare(counts[keep], q * T).pvalue > 1e-4
        np.testing.assert_allclose(logp, np.log(p)[tok], rtol=0, atol=1e-12)
    t1, l1, _, _ = oracle.sample_tokens_top_p(H[:2000], W, ones[:2000], 0.7, 1.0, seed=9, offset=3)
    t2, l2, _ = oracle.sample_tokens(H[:2000], W, ones[:2000], 0.7, seed=9, offset=3)
    np.testing.assert_array_equal(t1, t2)
    np.testing.assert_allclose(l1, l2, rtol=0, atol=1e-12)
    tok, _, _, _ = oracle.sample_tokens_top_p(H[:50], W, ones[:50], 1.0, 1e-9, seed=5, offset=0)
    assert np.all(tok == np.argmax(z))


def _nucleus_threshold_by_search(y, mass):
    """The nucleus threshold for a target mass: the highest distinct logit
    whose upper set carries at least `mass` of softmax(y) (explicit sums);
    the lowest logit when no threshold reaches it."""
    p = [math.exp(v) for v in y]
    total = math.fsum(p)
    for thr in sorted(set(y), reverse=True):
        if math.fsum(pv for pv, v in zip(p, y) if v >= thr) / total >= mass:
            return thr
    return min(y)


def test_top_p_band_brackets_the_nucleus_threshold():
    """The band sample_tokens_top_p returns for a row is [thr(top_p + band_mass)
    - band_logit, thr(top_p - band_mass) + band_logit], with thr(.) the
    nucleus threshold at that mass found by the explicit threshold search: so
    it contains the nucleus threshold at top_p itself, and is no wider than the
    mass and logit margins make it.  Rows with continuous logits and rows with
    many ties."""
    rng = np.random.default_rng(41)
    checked = 0
    for case in range(60):
        V, Hd = int(rng.integers(2, 40)), 4
        W = rng.normal(0, 1.0, (V, Hd))
        if case % 3 == 0:
            W = np.round(W * 2) / 2    # ties between vocabulary rows
        H = rng.normal(0, 1.0, (3, Hd))
        tau = float(rng.choice([0.7, 1.0, 1.5]))
        top_p = float(rng.uniform(0.05, 0.98))
        band_mass = float(rng.choice([1e-5, 1e-3, 0.05]))
        band_logit = float(rng.choice([0.0, 1e-4, 1e-2]))
        _, _, _, band = oracle.sample_tokens_top_p(H, W, np.ones(3, np.uint8), tau, top_p, seed=3, offset=case,
                                                   band_mass=band_mass, band_logit=band_logit)
        for t in range(3):
            y = ((W @ H[t]) / tau).tolist()
            lo = _nucleus_threshold_by_search(y, top_p + band_mass) - band_logit
            hi = _nucleus_threshold_by_search(y, top_p - band_mass) + band_logit
            assert band[t, 0] == pytest.approx(lo, rel=0, abs=1e-12), (case, t)
            assert band[t, 1] == pytest.approx(hi, rel=0, abs=1e-12), (case, t)
            thr = _nucleus_threshold_by_search(y, top_p)
            assert lo <= thr <= hi
            checked += 1
    assert checked == 180
    # top_p = 1 keeps everything: no band
    _, _, _, band = oracle.sample_tokens_top_p(np.ones((2, 3)), np.eye(3), np.ones(2, np.uint8), 1.0, 1.0, 1, 0)
    assert np.all(band == -np.inf)


# ---------------------------------------------------------------------------
# planted mistakes: each must trip one of the pins above
# ---------------------------------------------------------------------------

def test_planted_population_std_is_caught(monkeypatch):
    real = go.group_advantages
    monkeypatch.setattr(go, "group_advantages", lambda r, G, eps=1e-6, ddof=1: real(r, G, eps, ddof=0))
    monkeypatch.setattr(oracle, "group_advantages", go.group_advantages)
    with pytest.raises(AssertionError):
        test_advantage_closed_forms()


def test_planted_kl_without_minus_one_is_caught(monkeypatch):
    real = go.token_terms

    def bad(logp, old, ref, A, clip_eps, beta, *rest):
        tt = real(logp, old, ref, A, clip_eps, beta, *rest)
        tt["kl"] = tt["kl"] + 1.0
        tt["ell"] = -tt["s"] + beta * tt["kl"]
        return tt
    monkeypatch.setattr(go, "token_terms", bad)
    monkeypatch.setattr(oracle, "token_terms", bad)
    with pytest.raises(AssertionError):
        test_ratio_one_and_kl_zero_closed_forms()


def test_planted_target_off_by_one_is_caught(monkeypatch):
    real = go.token_logprobs
    monkeypatch.setattr(oracle, "token_logprobs",
                        lambda H, W, y, m, **kw: real(H, W, (np.asarray(y) + 1) % np.asarray(W).shape[0], m, **kw))
    with pytest.raises(AssertionError):
        test_logprobs_match_bruteforce_and_scipy()


def test_planted_gradient_sign_is_caught(monkeypatch):
    real = go.logp_coef

    def bad(logp, old, ref, A, w, clip_eps, beta, *rest):
        lp = np.asarray(logp, np.float64)
        tt = go.token_terms(logp, old, ref, A, clip_eps, beta)
        dsurr = np.where(tt["unclipped"], np.asarray(A) * tt["rho"], 0.0)
        return np.asarray(w) * (-dsurr - beta * (1.0 - np.exp(np.asarray(ref) - lp)))  # KL sign flipped
    monkeypatch.setattr(go, "logp_coef", bad)
    with pytest.raises(AssertionError):
        test_gradient_matches_central_differences(0)
    monkeypatch.setattr(go, "logp_coef", real)


def test_planted_clamp_without_gradient_cut_is_caught(monkeypatch):
    real = go.logp_coef
    # the capped tokens keep their KL gradient: the value is capped, the slope is not
    monkeypatch.setattr(go, "logp_coef", lambda *a: real(*a[:7]))
    with pytest.raises(AssertionError):
        test_clamped_kl_gradient_matches_central_differences()
    monkeypatch.setattr(go, "logp_coef", real)


def test_planted_adam_bias_correction_is_caught(monkeypatch):
    def bad(theta, m, v, g, lr, beta1, beta2, eps, weight_decay, step):
        m1 = beta1 * m + (1 - beta1) * g
        v1 = beta2 * v + (1 - beta2) * g * g
        return theta * (1 - lr * weight_decay) - lr * m1 / (np.sqrt(v1) + eps), m1, v1  # no bias correction
    monkeypatch.setattr(oracle, "adamw_step", bad)
    with pytest.raises(AssertionError):
        test_adamw_first_step_closed_form()


def test_planted_gumbel_sign_is_caught(monkeypatch):
    real = go.gumbel_noise
    monkeypatch.setattr(go, "gumbel_noise", lambda *a, **k: -real(*a, **k))
    with pytest.raises(AssertionError):
        test_gumbel_max_samples_follow_the_softmax()


def test_planted_nucleus_that_splits_ties_is_caught(monkeypatch):
    def bad(y, top_p):
        # the shortest prefix in stable order, ties with its last token cut off
        y = np.asarray(y, dtype=np.float64)
        if top_p >= 1.0:
            return np.ones(y.size, dtype=bool), -np.inf, 1.0
        p = scipy.special.softmax(y)
        order = np.argsort(-y, kind="stable")
        k = min(int(np.searchsorted(np.cumsum(p[order]), top_p, side="left")), y.size - 1)
        keep = np.zeros(y.size, dtype=bool)
        keep[order[:k + 1]] = True
        return keep, y[order[k]], float(p[keep].sum())
    monkeypatch.setattr(oracle, "nucleus", bad)
    with pytest.raises(AssertionError):
        test_nucleus_matches_threshold_search()


def test_planted_nucleus_one_token_too_many_is_caught(monkeypatch):
    real = go.nucleus

    def bad(y, top_p):
        keep, thr, mass = real(y, top_p)
        if top_p < 1.0 and not keep.all():
            y = np.asarray(y, dtype=np.float64)
            nxt = y[~keep].max()
            keep = y >= nxt
            thr = nxt
        return keep, thr, mass
    monkeypatch.setattr(oracle, "nucleus", bad)
    with pytest.raises(AssertionError):
        test_nucleus_matches_threshold_search()


def test_planted_widened_top_p_band_is_caught(monkeypatch):
    """A band ten times wider than its margins would excuse GPU/oracle
    disagreements it should not: the band pin must catch it."""
    real = go.sample_tokens_top_p

    def wide(*a, band_mass=1e-5, band_logit=1e-3, **kw):
        return real(*a, band_mass=10 * band_mass, band_logit=10 * band_logit, **kw)
    monkeypatch.setattr(oracle, "sample_tokens_top_p", wide)
    with pytest.raises(AssertionError):
        test_top_p_band_brackets_the_nucleus_threshold()


def test_planted_swapped_top_p_band_ends_are_caught(monkeypatch):
    """Band ends taken from the wrong side of top_p (the mass margins swapped)."""
    real = go.sample_tokens_top_p

    def swapped(*a, band_mass=1e-5, **kw):
        return real(*a, band_mass=-band_mass, **kw)
    monkeypatch.setattr(oracle, "sample_tokens_top_p", swapped)
    with pytest.raises(AssertionError):
        test_top_p_band_brackets_the_nucleus_threshold()
