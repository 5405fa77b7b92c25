"""GPU parity at the full 8B-shaped sizes (hidden 4096, vocabulary 155136),
in the launch configuration bench.py times (workspaces sized for the
unmasked rows).

The float64 oracle's log-sum-exp of every unmasked token (and the old /
reference log-probs, which are inputs of the loss) were written once by
tests/golden/make_golden.py, which calls only oracle/.  From them:

* logp: every token, |dlogp| <= 2e-3;
* loss: exact oracle loss over all tokens (O(T) from the stored values);
* dH: sampled rows the oracle computes one by one (full vocabulary sweep);
* dW: sampled vocabulary rows (a sum over all tokens), plus the invariant
  sum_v dW[v, :] = 0 on the whole GPU output.
"""
import os

import numpy as np
import pytest

import oracle
import workloads as wl
from tests._util import GRAD_RTOL, LOGP_ATOL, LOSS_RTOL, dev_tensor, loss_scale, near_clip_kink, rel_fro

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2507_05687_gb300 as grpo  # noqa: E402
from paper_2507_05687_gb300 import build as build_mod  # noqa: E402

build_mod.build()
DEV = torch.device("cuda", 0)
GOLDEN_DIR = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
BATCH = {"logprob3_8b": "batch8b", "fwdbwd_8b": "batch8b", "long_8b": "long_8b", "ragged_8b": "ragged_8b"}


def _load(name):
    path = os.path.join(GOLDEN_DIR, BATCH[name] + ".npz")
    if not os.path.exists(path):
        pytest.skip(f"stored oracle values {path} not generated")
    return np.load(path)


def _inputs(w, gold):
    Hb, Wb, y, m = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_targets(w), wl.gen_mask(w)
    idx = wl.valid_index(m)
    # the regenerated inputs must be the ones the stored values were computed on
    assert idx.size == int(gold["n_valid"])
    assert np.uint64(Hb[idx].astype(np.uint64).sum()) == gold["ck_h"]
    assert np.uint64(Wb.astype(np.uint64).sum()) == gold["ck_w"]
    assert np.uint64(y[idx].astype(np.uint64).sum()) == gold["ck_y"]
    return Hb, Wb, y, m, idx


def _target_logits(Hb, Wb, y, idx, chunk=16384):
    """z_{t, y_t} = H_t . W_{y_t} in float64 for the listed rows."""
    out = np.empty(idx.size)
    for a in range(0, idx.size, chunk):
        rows = idx[a:a + chunk]
        out[a:a + chunk] = np.einsum("ij,ij->i", oracle.widen_bf16(Hb[rows]), oracle.widen_bf16(Wb[y[rows]]))
    return out


def _oracle_logp(Hb, Wb, y, idx, lse):
    return _target_logits(Hb, Wb, y, idx) - lse


def test_logprob_three_heads_full_size():
    """Config: 8 prompts x G=8 x 512 tokens, policy / old / reference heads."""
    w = wl.WORKLOADS["logprob3_8b"]
    gold = _load(w.name)
    Hb, Wb, y, m, idx = _inputs(w, gold)
    H, yd, md = dev_tensor(Hb, torch.bfloat16), dev_tensor(y, torch.int32), dev_tensor(m, torch.uint8)
    ws = grpo.workspace(w.T, w.Hd, w.V, grpo.GRPO_WS_LOGPROBS, DEV, max_valid=idx.size)
    want = {"policy": _oracle_logp(Hb, Wb, y, idx, gold["lse_policy"]),
            "old": gold["old_logp"].astype(np.float64), "ref": gold["ref_logp"].astype(np.float64)}
    heads = []
    for which in ("policy", "old", "ref"):
        Wx = dev_tensor(Wb if which == "policy" else wl.gen_weight(w, which, Wb), torch.bfloat16)
        heads.append(Wx)
        lp = grpo.token_logprobs(H, Wx, yd, md, ws=ws)
        assert grpo.check_device_status(ws) == grpo.GRPO_OK
        got = lp.cpu().numpy()
        assert np.all(got[m == 0] == 0.0)
        err = np.abs(got[idx].astype(np.float64) - want[which])
        assert err.max() <= LOGP_ATOL, (which, err.max())
    # the three heads in one call (the configuration bench.py times for this workload)
    ws3 = grpo.workspace(w.T, w.Hd, w.V, grpo.GRPO_WS_LOGPROBS_HEADS, DEV, max_valid=idx.size)
    lp3 = grpo.token_logprobs_heads(H, heads, yd, md, ws=ws3)
    assert grpo.check_device_status(ws3) == grpo.GRPO_OK
    for h, which in enumerate(("policy", "old", "ref")):
        err = np.abs(lp3[h].cpu().numpy()[idx].astype(np.float64) - want[which])
        assert err.max() <= LOGP_ATOL, (which, err.max())


def _sample_rows(w, m, idx, r, k=96, skip=None):
    """Sampled compacted positions: first/last tokens, shortest and longest
    responses, zero-std groups, plus a seeded random draw; rows marked in
    `skip` (whose gradient is not unique at the log-prob tolerance) are left out."""
    lens = m.reshape(w.n_resp, w.L).sum(1)
    must = [idx[0], idx[-1]]
    for i in (int(np.argmin(lens)), int(np.argmax(lens))):
        must += [i * w.L, i * w.L + lens[i] - 1]
    zs = np.flatnonzero(r.reshape(w.n_prompts, w.G).std(1) == 0)
    for g in zs[:2]:
        must.append(g * w.G * w.L)
    pos = wl.sample_rows(idx.size, k, w.seed)
    rows = np.unique(np.concatenate([idx[pos], np.array(must, dtype=np.int64)]))
    rows = rows[m[rows] != 0]
    return rows if skip is None else rows[~skip[rows]]


_EXPECTED = {}   # per workload: the oracle's loss and its scale, sampled rows and their dH / dW rows
_PLAIN = {}      # per workload: the recomputing backward's (loss, dH, dW) on the device


def _expected(name, w, gold, Hb, Wb, y, m, idx, r, old, ref, adv):
    """The oracle's values the full-size checks compare against (computed once per workload)."""
    if name in _EXPECTED:
        return _EXPECTED[name]
    lse = np.zeros(w.T)
    lse[idx] = gold["lse_policy"]
    logp = np.zeros(w.T)
    logp[idx] = _oracle_logp(Hb, Wb, y, idx, gold["lse_policy"])
    want_loss, g, tt = oracle.grpo_loss(logp, old, ref, adv, m, w.n_resp, w.L, w.clip_eps, w.beta, 0)
    scale = loss_scale(want_loss, tt["w"], tt["ell"])
    # dH on sampled rows away from the clip kink, where the gradient is not unique
    rows = _sample_rows(w, m, idx, r, skip=near_clip_kink(logp, old, w.clip_eps) & (m != 0))
    want_dH = oracle.dH_rows(Hb, Wb, y, lse, g, rows)
    # dW on sampled vocabulary rows (target hits included)
    vrows = wl.sample_rows(w.V, 48, w.seed + 2, must=np.concatenate([[0, w.V - 1], y[idx[:16]]]))
    want_dW = oracle.dW_rows(Hb, Wb, y, m, lse, g, vrows)
    _EXPECTED[name] = dict(loss=want_loss, scale=scale, rows=rows, dH=want_dH, vrows=vrows, dW=want_dW)
    return _EXPECTED[name]


@pytest.mark.parametrize("name,kind", [(n, k) for n in ("fwdbwd_8b", "long_8b", "ragged_8b")
                                       for k in ("plain", "kept")])
def test_fwd_bwd_full_size(name, kind):
    """plain: the default backward, which recomputes each vocabulary chunk of
    the logits (no [tokens x vocabulary] buffer), against the oracle.  kept:
    the opt-in backward that stores the forward's logits, against the oracle
    and bit for bit against the plain one.  Workspaces as bench.py sizes them
    (for the unmasked rows)."""
    w = wl.WORKLOADS[name]
    gold = _load(name)
    Hb, Wb, y, m, idx = _inputs(w, gold)
    r = wl.gen_rewards(w)
    old = np.zeros(w.T, np.float32)
    ref = np.zeros(w.T, np.float32)
    old[idx], ref[idx] = gold["old_logp"], gold["ref_logp"]
    adv = oracle.group_advantages(r, w.G, float(np.float32(w.adv_eps)))
    want = _expected(name, w, gold, Hb, Wb, y, m, idx, r, old, ref, adv)

    H, W = dev_tensor(Hb, torch.bfloat16), dev_tensor(Wb, torch.bfloat16)
    cap = (idx.size + 255) // 256 * 256
    which = grpo.GRPO_WS_LOSS if kind == "plain" else grpo.GRPO_WS_LOSS_LOGITS
    ws = grpo.workspace(w.T, w.Hd, w.V, which, DEV, max_valid=idx.size)
    assert grpo.loss_plan(w.T, w.Hd, w.V, ws.numel()) == (int(kind == "kept"), cap)
    adv_d = grpo.group_advantages(dev_tensor(r, torch.float32), w.G, w.adv_eps)
    assert np.array_equal(adv_d.cpu().numpy().view(np.uint32), adv.view(np.uint32))
    loss, dH, dW = grpo.loss_fwd_bwd(H, W, dev_tensor(y, torch.int32), dev_tensor(m, torch.uint8),
                                     dev_tensor(old, torch.float32), dev_tensor(ref, torch.float32), adv_d,
                                     w.n_resp, w.L, w.clip_eps, w.beta, 0, ws=ws)
    assert grpo.check_device_status(ws) == grpo.GRPO_OK
    del ws

    # loss over every token, from the stored oracle log-sum-exp: the bar on
    # max(|loss|, sum_t |w_t l_t|), and the plain relative error reported
    d = abs(loss.item() - want["loss"])
    print(f"[{name}-{kind}] loss {loss.item():.9g} oracle {want['loss']:.9g} rel {d / abs(want['loss']):.3g} "
          f"rel_terms {d / want['scale']:.3g}")
    assert d <= LOSS_RTOL * want["scale"], (loss.item(), want["loss"], want["scale"])

    got_dH = dH[torch.from_numpy(want["rows"]).to(DEV)].double().cpu().numpy()
    assert rel_fro(got_dH, want["dH"]) <= GRAD_RTOL, rel_fro(got_dH, want["dH"])
    pad = np.flatnonzero(m == 0)
    if pad.size:   # padding rows exactly zero
        pr = pad[wl.sample_rows(pad.size, 256, w.seed + 1)]
        assert not dH[torch.from_numpy(pr).to(DEV)].any()
    got_dW = dW[torch.from_numpy(want["vrows"]).to(DEV)].double().cpu().numpy()
    assert rel_fro(got_dW, want["dW"]) <= GRAD_RTOL, rel_fro(got_dW, want["dW"])

    # sum_v dZ_{t,v} = 0 for every token, hence the columns of dW sum to ~0
    colsum = dW.double().sum(0)
    colabs = dW.double().abs().sum(0)
    assert (colsum.norm() / colabs.norm()).item() <= 1e-2

    if kind == "plain":
        _PLAIN[name] = (loss, dH, dW)
    else:
        plain = _PLAIN.pop(name, None)
        if plain is not None:   # the two backwards give the same bits
            for a, b in zip((loss, dH, dW), plain):
                assert torch.equal(a, b)
        del plain
        torch.cuda.empty_cache()


def test_sampling_full_size():
    """The rollout draw over the 32768-row batch at 4096 x 155136, checked on sampled rows."""
    w = wl.WORKLOADS["logprob3_8b"]
    Hb, Wb, m = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_mask(w)
    ws = grpo.workspace(w.T, w.Hd, w.V, grpo.GRPO_WS_SAMPLE, DEV, max_valid=int(m.sum()))
    tok, lp = grpo.sample_tokens(dev_tensor(Hb, torch.bfloat16), dev_tensor(Wb, torch.bfloat16),
                                 dev_tensor(m, torch.uint8), 1.0, seed=20250705, offset=687, ws=ws)
    tok, lp = tok.cpu().numpy(), lp.cpu().numpy()
    assert np.all(tok[m == 0] == -1)
    idx = wl.valid_index(m)
    assert tok[idx].min() >= 0 and tok[idx].max() < w.V
    rows = idx[wl.sample_rows(idx.size, 96, w.seed + 5)]
    want_tok, want_lp, gap = oracle.sample_tokens(Hb, Wb, m, 1.0, 20250705, 687, rows=rows)
    clear = rows[gap[rows] > 1e-3]
    assert clear.size >= 0.9 * rows.size
    assert np.array_equal(tok[clear], want_tok[clear])
    assert np.abs(lp[clear] - want_lp[clear]).max() <= LOGP_ATOL


def test_decode_step_full_vocabulary():
    """One decode step of 256 sequences at 4096 x 155136 (forward units narrowed
    to 8 vocabulary tiles, 76 splits): every row's log-prob against the oracle's
    float64 log-sum-exp, and every row's draw against the oracle's Gumbel-max."""
    w = wl.DECODE_WORKLOADS["decode256_8b"]
    Hb, Wb, y, m = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_targets(w), wl.gen_mask(w)
    H, W = dev_tensor(Hb, torch.bfloat16), dev_tensor(Wb, torch.bfloat16)
    got = grpo.token_logprobs(H, W, dev_tensor(y, torch.int32), dev_tensor(m, torch.uint8)).cpu().numpy()
    want, _ = oracle.token_logprobs(Hb, Wb, y, m)
    assert np.abs(got.astype(np.float64) - want).max() <= LOGP_ATOL
    tok, lp = grpo.sample_tokens(H, W, dev_tensor(m, torch.uint8), 0.7, seed=9, offset=2**33 + 5)
    tok, lp = tok.cpu().numpy(), lp.cpu().numpy()
    want_tok, want_lp, gap = oracle.sample_tokens(Hb, Wb, m, 0.7, 9, 2**33 + 5)
    clear = np.flatnonzero(gap > 1e-3)
    assert clear.size >= 0.9 * w.T
    assert np.array_equal(tok[clear], want_tok[clear])
    assert np.abs(lp[clear] - want_lp[clear]).max() <= LOGP_ATOL
