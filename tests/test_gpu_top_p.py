"""The rollout draw restricted to the nucleus (grpo_sample_tokens_top_p)
against the oracle's nucleus sampler on the same Philox noise.

The GPU decides the nucleus from fp32 logits and fp32 probabilities summed in
fixed point, the oracle in fp64 with a sort.  A draw may differ only where the
oracle's best perturbed score beats the second by at most 2e-3, or where the
GPU's or the oracle's token lies in the oracle's boundary band (logits whose
membership changes if the cumulative masses move by band_mass or the logits by
band_logit); at least 90% of the rows must agree exactly.
"""
import numpy as np
import pytest
import scipy.special

import oracle
import workloads as wl
from tests._util import LOGP_ATOL, dev_tensor

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2507_05687_gb300 as grpo  # noqa: E402
from paper_2507_05687_gb300 import build as build_mod  # noqa: E402

build_mod.build()
DEV = torch.device("cuda", 0)
TIE = 2e-3


def _draw(Hb, Wb, m, tau, top_p, seed, offset, ws=None):
    tok, lp = grpo.sample_tokens_top_p(dev_tensor(Hb, torch.bfloat16), dev_tensor(Wb, torch.bfloat16),
                                       dev_tensor(m, torch.uint8), tau, top_p, seed=seed, offset=offset, ws=ws)
    return tok.cpu().numpy(), lp.cpu().numpy()


def _compare(Hb, Wb, m, tau, top_p, seed, offset, tok, logp, band_mass=1e-5, band_logit=1e-4, rows=None):
    want, want_lp, gap, band = oracle.sample_tokens_top_p(Hb, Wb, m, tau, top_p, seed, offset, rows=rows,
                                                           band_mass=band_mass, band_logit=band_logit)
    idx = wl.valid_index(m) if rows is None else np.asarray(rows)
    assert np.all(tok[m == 0] == -1) and np.all(logp[m == 0] == 0.0)
    same = tok[idx] == want[idx]
    assert same.mean() >= 0.9, same.mean()
    Wf = oracle.as_f64(Wb)
    for t in idx:
        h = oracle.as_f64(Hb[t])
        y_got, y_want = (h @ Wf[tok[t]]) / tau, (h @ Wf[want[t]]) / tau
        lo, hi = band[t]
        assert y_got >= lo, (t, y_got, lo)         # never outside the nucleus and its band
        if tok[t] != want[t]:
            in_band = lo <= y_got <= hi or lo <= y_want <= hi
            assert gap[t] <= TIE or in_band, (t, tok[t], want[t], gap[t])
    ok = idx[same]
    assert np.abs(logp[ok] - want_lp[ok]).max() <= LOGP_ATOL
    return same.mean()


@pytest.mark.parametrize("tau,top_p,w_std,V", [(1.0, 0.9, 0.08, 5000), (0.7, 0.5, 0.08, 4097),
                                               (1.0, 0.95, 0.6, 5000), (1.6, 0.3, 0.3, 3000)])
def test_top_p_matches_oracle(tau, top_p, w_std, V):
    """Flat (w_std 0.08: most of the vocabulary in the nucleus) and peaked
    (0.3-0.6: a few tokens) distributions, ragged rows, vocabulary tails."""
    w = wl.Workload("p", 2, 3, 90, 192, V, "uniform", 1, 90, seed=wl.SEED_BASE + 2600 + V, w_std=w_std)
    Hb, Wb, m = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_mask(w)
    tok, lp = _draw(Hb, Wb, m, tau, top_p, 2507, 19)
    _compare(Hb, Wb, m, tau, top_p, 2507, 19, tok, lp)


def test_top_p_one_is_the_plain_sampler():
    """top_p = 1 keeps the whole vocabulary: the same tokens and log-probs as
    grpo_sample_tokens bit for bit (same noise, same fp32 operations, the same
    merge of the vocabulary splits)."""
    w = wl.Workload("p", 2, 4, 70, 256, 4500, "uniform", 1, 70, seed=wl.SEED_BASE + 2700, w_std=0.1)
    Hb, Wb, m = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_mask(w)
    H, W, md = dev_tensor(Hb, torch.bfloat16), dev_tensor(Wb, torch.bfloat16), dev_tensor(m, torch.uint8)
    for tau in (1.0, 0.8):
        a_tok, a_lp = grpo.sample_tokens_top_p(H, W, md, tau, 1.0, seed=5, offset=77)
        b_tok, b_lp = grpo.sample_tokens(H, W, md, tau, seed=5, offset=77)
        assert torch.equal(a_tok, b_tok) and torch.equal(a_lp, b_lp)


def test_tiny_top_p_is_greedy():
    w = wl.Workload("p", 1, 4, 60, 128, 3000, "uniform", 1, 60, seed=wl.SEED_BASE + 2800, w_std=0.3)
    Hb, Wb, m = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_mask(w)
    tok, _ = _draw(Hb, Wb, m, 1.0, 1e-7, 3, 0)
    idx = wl.valid_index(m)
    Z = oracle.as_f64(Hb[idx]) @ oracle.as_f64(Wb).T
    top2 = np.sort(Z, axis=1)[:, -2:]
    clear = top2[:, 1] - top2[:, 0] > 1e-3
    assert clear.mean() > 0.9
    assert np.array_equal(tok[idx][clear], np.argmax(Z, axis=1)[clear])


def test_top_p_frequencies_follow_the_truncated_softmax():
    """20000 rows with the same logits over 7 tokens: inside the nucleus the
    frequencies follow the renormalised softmax, outside they are zero."""
    from scipy.stats import chisquare
    Hd, V, T = 64, 7, 20000
    rng = np.random.default_rng(3)
    Wb = wl.f32_to_bf16_bits(rng.normal(0, 0.15, (V, Hd)).astype(np.float32))
    hb = wl.f32_to_bf16_bits(rng.normal(0, 1, Hd).astype(np.float32))
    z = oracle.as_f64(Wb) @ oracle.as_f64(hb)
    H = dev_tensor(np.tile(hb, (T, 1)), torch.bfloat16)
    md = torch.ones(T, dtype=torch.uint8, device=DEV)
    for tau, top_p in ((1.0, 0.9), (2.0, 0.8), (0.5, 0.9)):   # nuclei of 4, 5 and 2 of the 7 tokens
        keep = oracle.nucleus(z / tau, top_p)[0]
        assert 1 < keep.sum() < V
        tok = grpo.sample_tokens_top_p(H, dev_tensor(Wb, torch.bfloat16), md, tau, top_p, seed=77,
                                       offset=3)[0].cpu().numpy()
        counts = np.bincount(tok, minlength=V)
        assert counts[~keep].sum() == 0
        p = scipy.special.softmax(z / tau)[keep]
        assert chisquare(counts[keep], p / p.sum() * T).pvalue > 1e-4


def test_tied_logits_at_the_boundary_stay_together():
    """Two identical LM-head rows give exactly equal logits; with the nucleus
    boundary on them both are drawn (about equally often) and nothing below."""
    Hd, V, T = 64, 6, 20000
    rng = np.random.default_rng(11)
    hb = wl.f32_to_bf16_bits(rng.normal(0, 1, Hd).astype(np.float32))
    h = oracle.as_f64(hb)
    # rows scaled along h so that the logits are about (2.0, 1.0, 1.0, 0.0, -1.0, -2.0)
    base = wl.f32_to_bf16_bits((h / (h @ h)).astype(np.float32))
    Wf = np.stack([oracle.as_f64(base) * c for c in (2.0, 1.0, 1.0, 0.0, -1.0, -2.0)]).astype(np.float32)
    Wb = wl.f32_to_bf16_bits(Wf)
    Wb[2] = Wb[1]                                   # an exact tie
    z = oracle.as_f64(Wb) @ h
    p = scipy.special.softmax(z)
    top_p = float(p[0] + 0.5 * p[1])                # the boundary falls on the tied pair
    keep = oracle.nucleus(z, top_p)[0]
    assert keep.tolist() == [True, True, True, False, False, False]
    H = dev_tensor(np.tile(hb, (T, 1)), torch.bfloat16)
    md = torch.ones(T, dtype=torch.uint8, device=DEV)
    tok = grpo.sample_tokens_top_p(H, dev_tensor(Wb, torch.bfloat16), md, 1.0, top_p, seed=8, offset=1)[0]
    counts = np.bincount(tok.cpu().numpy(), minlength=V)
    assert counts[3:].sum() == 0
    assert counts[1] > 0.4 * counts[1:3].sum() and counts[2] > 0.4 * counts[1:3].sum()


def test_crowded_bucket_is_refined():
    """A narrow logit spread puts more than 1024 logits in the bucket that
    holds the threshold: the kernel refines that bucket (a second histogram
    over its own range) before resolving the candidates; all-equal logits are
    taken whole (the plain sampler's draw)."""
    w = wl.Workload("p", 1, 2, 40, 64, 50000, "uniform", 1, 40, seed=wl.SEED_BASE + 2900, w_std=0.018)
    Hb, Wb, m = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_mask(w)
    idx = wl.valid_index(m)
    Z = oracle.as_f64(Hb[idx[0]]) @ oracle.as_f64(Wb).T
    y_thr = oracle.nucleus(Z, 0.5)[1]
    bucket = np.floor((Z.max() - Z) * 64)           # the kernel's first-level buckets (1/64 nat)
    assert np.sum(bucket == np.floor((Z.max() - y_thr) * 64)) > 1024
    tok, lp = _draw(Hb, Wb, m, 1.0, 0.5, 41, 2)
    _compare(Hb, Wb, m, 1.0, 0.5, 41, 2, tok, lp, band_mass=2e-6, band_logit=1e-5)
    # all logits equal (W = 0): every token is in the nucleus
    H, W0 = dev_tensor(Hb, torch.bfloat16), torch.zeros(5000, 64, dtype=torch.bfloat16, device=DEV)
    md = dev_tensor(m, torch.uint8)
    a = grpo.sample_tokens_top_p(H, W0, md, 1.0, 0.3, seed=4, offset=0)[0]
    b = grpo.sample_tokens(H, W0, md, 1.0, seed=4, offset=0)[0]
    assert torch.equal(a, b)


def test_top_p_lean_workspace_capacity_and_arguments():
    w = wl.Workload("p", 2, 4, 100, 128, 1500, "uniform", 1, 30, seed=wl.SEED_BASE + 3000, w_std=0.2)
    Hb, Wb, m = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_mask(w)
    nv = int(m.sum())
    assert nv <= 256 < w.T
    full = _draw(Hb, Wb, m, 1.0, 0.8, 6, 6)
    ws = grpo.workspace(w.T, w.Hd, w.V, grpo.GRPO_WS_SAMPLE_TOP_P, DEV, max_valid=nv)
    assert ws.numel() < grpo.workspace_bytes(w.T, w.Hd, w.V, grpo.GRPO_WS_SAMPLE_TOP_P)
    lean = _draw(Hb, Wb, m, 1.0, 0.8, 6, 6, ws=ws)
    assert grpo.check_device_status(ws) == grpo.GRPO_OK
    assert np.array_equal(full[0], lean[0]) and np.array_equal(full[1], lean[1])
    # every row unmasked: 800 rows against a capacity of 256
    allm = np.ones_like(m)
    tok, _ = _draw(Hb, Wb, allm, 1.0, 0.8, 6, 6, ws=ws)
    assert grpo.check_device_status(ws) == grpo.GRPO_ERR_CAPACITY
    assert np.all(tok[256:] == -1)
    H, W = dev_tensor(Hb, torch.bfloat16), dev_tensor(Wb, torch.bfloat16)
    md = dev_tensor(m, torch.uint8)
    for bad in (0.0, -0.1, 1.5, float("nan")):
        with pytest.raises(grpo.GrpoError):
            grpo.sample_tokens_top_p(H, W, md, 1.0, bad)
    empty = grpo.sample_tokens_top_p(H[:0], W, md[:0], 1.0, 0.9)
    assert empty[0].numel() == 0


@pytest.mark.parametrize("top_p,n_rows", [(0.9, 256), (0.5, 128)])
def test_top_p_decode_step_full_vocabulary(top_p, n_rows):
    """A decode step of the 8B head (256 rows x 155,136 tokens, Hd 4096)
    against the oracle (on n_rows of the rows): the shape the nucleus draw
    serves in rollout generation, with about (1 - top_p) of the rows through
    the cluster kernel's histogram path."""
    w = wl.DECODE_WORKLOADS["decode256_8b"]
    Hb, Wb, m = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_mask(w)
    tok, lp = _draw(Hb, Wb, m, 1.0, top_p, 20250705, 9)
    _compare(Hb, Wb, m, 1.0, top_p, 20250705, 9, tok, lp, rows=wl.valid_index(m)[:n_rows])
    # the order in which rows join the cluster kernel's list varies between
    # calls; the draws and their log-probs do not
    again = _draw(Hb, Wb, m, 1.0, top_p, 20250705, 9)
    assert np.array_equal(tok, again[0]) and np.array_equal(lp, again[1])


@pytest.mark.parametrize("V", [1, 2, 3, 5])
def test_top_p_tiny_vocabularies(V):
    """Vocabularies below and just above one 4-logit group: the walks' tails
    alone (and, at V = 1, a nucleus that is the single token)."""
    w = wl.Workload("p", 2, 4, 30, 64, V, "uniform", 1, 30, seed=wl.SEED_BASE + 3100 + V, w_std=0.5)
    Hb, Wb, m = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_mask(w)
    for top_p in (0.5, 0.9):
        tok, lp = _draw(Hb, Wb, m, 1.0, top_p, 12, 3)
        assert np.all(tok[m != 0] >= 0) and np.all(tok[m != 0] < V)
        _compare(Hb, Wb, m, 1.0, top_p, 12, 3, tok, lp)


@pytest.mark.parametrize("top_p", [0.3, 0.9])
def test_every_row_listed_gives_the_same_draws(monkeypatch, top_p):
    """The streaming pass lists only rows whose winner may lie outside the
    nucleus (from fp32 sums within a bound of the exact mass); the selection
    confirms each listed row with the exact mass and leaves a row whose mass
    above the winner falls short with its plain draw.  With every row listed
    (a test hook), that confirmation decides all of them: the draws and
    log-probs are the same bits as with the bound, on a flat and a peaked
    distribution and a decode step of the full vocabulary."""
    cases = [wl.Workload("p", 2, 3, 90, 192, 5000, "uniform", 1, 90, seed=wl.SEED_BASE + 3300, w_std=0.08),
             wl.Workload("p", 2, 3, 90, 192, 4097, "uniform", 1, 90, seed=wl.SEED_BASE + 3301, w_std=0.5),
             wl.DECODE_WORKLOADS["decode256_8b"]]
    for w in cases:
        Hb, Wb, m = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_mask(w)
        want = _draw(Hb, Wb, m, 1.0, top_p, 77, 5)
        monkeypatch.setenv("GRPO_TEST_TOP_P_LIST_ALL", "1")
        got = _draw(Hb, Wb, m, 1.0, top_p, 77, 5)
        monkeypatch.delenv("GRPO_TEST_TOP_P_LIST_ALL")
        assert np.array_equal(got[0], want[0]) and np.array_equal(got[1], want[1])


@pytest.mark.parametrize("top_p", [0.9, 0.5])
def test_cluster_size_gives_the_same_draws(monkeypatch, top_p):
    """The selection takes each listed row in a cluster of 16, 8, 4 or 2 CTAs
    (chosen by the expected number of listed rows); the histogram merge, the
    candidate split of the threshold search and the draw's entry split all
    change with the size, and every reduction in them is exact or has a total
    order, so the draws and log-probs are the same bits for every size, here
    with every row listed too (both levels of the selection run on every
    row) and on a crowded vocabulary that needs a second histogram level."""
    cases = [wl.Workload("p", 2, 3, 90, 192, 5000, "uniform", 1, 90, seed=wl.SEED_BASE + 3310, w_std=0.08),
             wl.Workload("p", 2, 3, 90, 192, 4097, "uniform", 1, 90, seed=wl.SEED_BASE + 3311, w_std=0.5),
             wl.Workload("p", 1, 2, 40, 64, 50000, "uniform", 1, 40, seed=wl.SEED_BASE + 2900, w_std=0.018),
             wl.DECODE_WORKLOADS["decode256_8b"]]
    for w in cases:
        Hb, Wb, m = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_mask(w)
        for list_all in ("0", "1"):
            monkeypatch.setenv("GRPO_TEST_TOP_P_LIST_ALL", list_all)
            got = {}
            for c in ("8", "16", "4", "2"):
                monkeypatch.setenv("GRPO_TOP_P_CLUSTER", c)
                got[c] = _draw(Hb, Wb, m, 1.0, top_p, 91, 3)
            for c in ("16", "4", "2"):
                assert np.array_equal(got[c][0], got["8"][0]) and np.array_equal(got[c][1], got["8"][1]), (w.V, c)
    monkeypatch.delenv("GRPO_TOP_P_CLUSTER")
    monkeypatch.delenv("GRPO_TEST_TOP_P_LIST_ALL")
