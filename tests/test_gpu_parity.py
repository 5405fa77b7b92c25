"""GPU parity of the CUDA path against the float64 oracle, element by element,
at sizes the oracle finishes in seconds: several tiles, ragged tails, several
vocabulary splits and backward chunks, and the degenerate cases."""
import numpy as np
import pytest

import oracle
import workloads as wl
from tests._util import GRAD_RTOL, LOGP_ATOL, LOSS_RTOL, clear_of_clip_kink, dev_tensor, loss_scale, rel_fro

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2507_05687_gb300 as grpo  # noqa: E402
from paper_2507_05687_gb300 import build as build_mod  # noqa: E402

build_mod.build()
DEV = torch.device("cuda", 0)


def _case(w, agg_mode=0):
    """Seeded inputs of workload w plus the oracle's outputs on them."""
    Hb, Wb = wl.gen_hidden(w), wl.gen_weight(w)
    y, m, r = wl.gen_targets(w), wl.gen_mask(w), wl.gen_rewards(w)
    W_old, W_ref = wl.gen_weight(w, "old", Wb), wl.gen_weight(w, "ref", Wb)
    old = oracle.token_logprobs(Hb, W_old, y, m)[0].astype(np.float32)
    old = clear_of_clip_kink(oracle.token_logprobs(Hb, Wb, y, m)[0], old, w.clip_eps)
    ref = oracle.token_logprobs(Hb, W_ref, y, m)[0].astype(np.float32)
    adv = oracle.group_advantages(r, w.G, float(np.float32(w.adv_eps)))
    want = oracle.loss_fwd_bwd(Hb, Wb, y, m, old, ref, adv, w.n_resp, w.L, w.clip_eps, w.beta, agg_mode)
    return dict(w=w, H=Hb, W=Wb, y=y, m=m, r=r, old=old, ref=ref, adv=adv, want=want)


def _dev(c):
    return dict(H=dev_tensor(c["H"], torch.bfloat16), W=dev_tensor(c["W"], torch.bfloat16),
                y=dev_tensor(c["y"], torch.int32), m=dev_tensor(c["m"], torch.uint8),
                old=dev_tensor(c["old"], torch.float32), ref=dev_tensor(c["ref"], torch.float32),
                adv=dev_tensor(c["adv"], torch.float32), r=dev_tensor(c["r"], torch.float32))


def _check_fwd_bwd(c, agg_mode=0, kind=grpo.GRPO_WS_LOSS):
    w, d = c["w"], _dev(c)
    ws = grpo.workspace(w.T, w.Hd, w.V, kind, DEV)
    assert grpo.loss_plan(w.T, w.Hd, w.V, ws.numel())[0] == (kind == grpo.GRPO_WS_LOSS_LOGITS)
    loss, dH, dW = grpo.loss_fwd_bwd(d["H"], d["W"], d["y"], d["m"], d["old"], d["ref"], d["adv"],
                                     w.n_resp, w.L, w.clip_eps, w.beta, agg_mode, ws=ws)
    assert grpo.check_device_status(ws) == grpo.GRPO_OK
    want = c["want"]
    scale = loss_scale(want["loss"], want["terms"]["w"], want["terms"]["ell"])
    assert abs(loss.item() - want["loss"]) <= LOSS_RTOL * scale, (loss.item(), want["loss"], scale)
    dHn, dWn = dH.double().cpu().numpy(), dW.double().cpu().numpy()
    assert rel_fro(dHn, want["dH"]) <= GRAD_RTOL, rel_fro(dHn, want["dH"])
    assert rel_fro(dWn, want["dW"]) <= GRAD_RTOL, rel_fro(dWn, want["dW"])
    assert np.all(dHn[c["m"] == 0] == 0.0)
    return loss, dH, dW


# ---------------------------------------------------------------- Eq. 2

@pytest.mark.parametrize("G", [2, 3, 4, 5, 8, 16, 32, 48, 64, 100])
def test_advantages_bit_exact_dyadic(G):
    rng = np.random.default_rng(G)
    r = (rng.integers(0, 5, size=G * 37) / 4.0).astype(np.float32)   # {0, .25, .5, .75, 1}
    r[:G] = 0.5                                                       # a zero-std group
    got = grpo.group_advantages(dev_tensor(r, torch.float32), G, 1e-6).cpu().numpy()
    want = oracle.group_advantages(r, G, float(np.float32(1e-6)))
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))


@pytest.mark.parametrize("G", [2, 7, 8, 32, 33])
def test_advantages_general_rewards_within_one_ulp(G):
    rng = np.random.default_rng(100 + G)
    r = rng.normal(size=G * 50).astype(np.float32)
    got = grpo.group_advantages(dev_tensor(r, torch.float32), G, 1e-6).cpu().numpy()
    want = oracle.group_advantages(r, G, float(np.float32(1e-6)))
    ulp = np.abs(got.view(np.int32).astype(np.int64) - want.view(np.int32).astype(np.int64))
    assert ulp.max() <= 1


@pytest.mark.parametrize("name", list(wl.WORKLOADS))
def test_advantages_of_every_workload_bit_exact(name):
    w = wl.WORKLOADS[name]
    r = wl.gen_rewards(w)
    got = grpo.group_advantages(dev_tensor(r, torch.float32), w.G, w.adv_eps).cpu().numpy()
    want = oracle.group_advantages(r, w.G, float(np.float32(w.adv_eps)))
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))


# ---------------------------------------------------------------- log-probs

LOGP_SHAPES = [
    # (n_prompts, G, L, Hd, V, lengths)
    (1, 4, 64, 256, 4096, "full"),            # the tiny workload's shape
    (2, 3, 150, 192, 1000, "uniform"),        # vocabulary tail (1000 = 3*256 + 232), ragged rows
    (1, 2, 65, 64, 300, "uniform"),           # one k-block, tail
    (3, 4, 97, 512, 8292, "uniform"),         # three vocabulary splits, tail of 100
]


@pytest.mark.parametrize("shape", LOGP_SHAPES)
def test_logprobs_match_oracle(shape):
    P, G, L, Hd, V, lens = shape
    w = wl.Workload("t", P, G, L, Hd, V, lens, 1, L, seed=wl.SEED_BASE + 1000 + Hd + V)
    Hb, Wb, y, m = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_targets(w), wl.gen_mask(w)
    want, _ = oracle.token_logprobs(Hb, Wb, y, m)
    got = grpo.token_logprobs(dev_tensor(Hb, torch.bfloat16), dev_tensor(Wb, torch.bfloat16),
                              dev_tensor(y, torch.int32), dev_tensor(m, torch.uint8)).cpu().numpy()
    assert np.all(got[m == 0] == 0.0)
    err = np.abs(got.astype(np.float64) - want)
    assert err.max() <= LOGP_ATOL, err.max()


@pytest.mark.parametrize("n_heads", [1, 2, 3, 4])
def test_logprobs_heads_match_oracle_and_single_calls(n_heads):
    """Policy / old / reference (and a fourth) heads in one call: each row matches
    the oracle, and the single-head call bit for bit."""
    w = wl.Workload("t", 2, 3, 120, 256, 4400, "uniform", 1, 120, seed=wl.SEED_BASE + 1500 + n_heads)
    Hb, Wb, y, m = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_targets(w), wl.gen_mask(w)
    heads = [Wb, wl.gen_weight(w, "old", Wb), wl.gen_weight(w, "ref", Wb), wl.gen_weight(w.with_(w_std=0.05))][:n_heads]
    H, yd, md = dev_tensor(Hb, torch.bfloat16), dev_tensor(y, torch.int32), dev_tensor(m, torch.uint8)
    Wd = [dev_tensor(x, torch.bfloat16) for x in heads]
    got = grpo.token_logprobs_heads(H, Wd, yd, md)
    assert got.shape == (n_heads, w.T)
    for h in range(n_heads):
        want, _ = oracle.token_logprobs(Hb, heads[h], y, m)
        g = got[h].cpu().numpy()
        assert np.all(g[m == 0] == 0.0)
        assert np.abs(g - want).max() <= LOGP_ATOL
        assert torch.equal(got[h], grpo.token_logprobs(H, Wd[h], yd, md))


def test_logprobs_large_logits_and_host_buffers():
    w = wl.Workload("t", 2, 2, 70, 128, 777, "uniform", 1, 70, seed=wl.SEED_BASE + 77, w_std=0.5)
    Hb, Wb, y, m = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_targets(w), wl.gen_mask(w)
    want, _ = oracle.token_logprobs(Hb, Wb, y, m)
    # CPU tensors in, CPU tensor out (host<->device copies inside the call)
    got = grpo.token_logprobs(torch.from_numpy(Hb).view(torch.bfloat16), torch.from_numpy(Wb).view(torch.bfloat16),
                              torch.from_numpy(y), torch.from_numpy(m))
    assert got.device.type == "cpu"
    assert np.abs(got.numpy() - want).max() <= LOGP_ATOL * 4  # logits ~ +-100 here


# ---------------------------------------------------------------- forward + backward

def test_tiny_workload_fwd_bwd():
    _check_fwd_bwd(_case(wl.WORKLOADS["tiny_fwdbwd"]))


@pytest.mark.parametrize("agg_mode", [0, 1])
def test_ragged_multi_chunk_fwd_bwd(agg_mode, monkeypatch):
    monkeypatch.setenv("GRPO_VOCAB_CHUNK", "512")   # several backward chunks + a tail chunk
    w = wl.Workload("t", 2, 4, 90, 320, 1800, "uniform", 1, 90, rewards="mix", seed=wl.SEED_BASE + 500)
    _check_fwd_bwd(_case(w, agg_mode), agg_mode)


@pytest.mark.parametrize("layout", ["rows", "blocks"])
def test_transposed_hidden_state_layouts(layout, monkeypatch):
    """dW reads the gathered hidden states transposed, as plain rows or in
    64-token k-blocks (chosen by length; forced here on a small ragged case)."""
    monkeypatch.setenv("GRPO_HCT_LAYOUT", layout)
    monkeypatch.setenv("GRPO_VOCAB_CHUNK", "768")
    w = wl.Workload("t", 3, 4, 60, 192, 2100, "uniform", 1, 60, rewards="mix", seed=wl.SEED_BASE + 560)
    _check_fwd_bwd(_case(w))


@pytest.mark.parametrize("pair", ["0", "1"])
def test_single_and_paired_tiles_agree(pair, monkeypatch):
    """The 128x256 single-CTA tile and the 256x256 CTA-pair tile both meet the bar."""
    monkeypatch.setenv("GRPO_CTA_PAIR", pair)
    monkeypatch.setenv("GRPO_VOCAB_CHUNK", "768")
    w = wl.Workload("t", 3, 4, 60, 192, 2100, "uniform", 1, 60, rewards="mix", seed=wl.SEED_BASE + 550)
    _check_fwd_bwd(_case(w))


@pytest.mark.parametrize("agg_mode", [0, 1])
def test_global_normaliser(agg_mode):
    """grpo_loss_fwd_bwd_norm: this batch as one shard of a larger data-parallel batch."""
    w = wl.Workload("t", 2, 4, 50, 128, 900, "uniform", 1, 50, rewards="mix", seed=wl.SEED_BASE + 650)
    c = _case(w, agg_mode)
    norm = 3.5 * (c["m"].sum() if agg_mode == 0 else w.n_resp)
    want = oracle.loss_fwd_bwd(c["H"], c["W"], c["y"], c["m"], c["old"], c["ref"], c["adv"], w.n_resp, w.L,
                               w.clip_eps, w.beta, agg_mode, norm=norm)
    d = _dev(c)
    loss, dH, dW = grpo.loss_fwd_bwd(d["H"], d["W"], d["y"], d["m"], d["old"], d["ref"], d["adv"], w.n_resp, w.L,
                                     w.clip_eps, w.beta, agg_mode, norm=norm)
    scale = loss_scale(want["loss"], want["terms"]["w"], want["terms"]["ell"])
    assert abs(loss.item() - want["loss"]) <= LOSS_RTOL * scale
    assert rel_fro(dH.double().cpu().numpy(), want["dH"]) <= GRAD_RTOL
    assert rel_fro(dW.double().cpu().numpy(), want["dW"]) <= GRAD_RTOL


@pytest.mark.parametrize("agg_mode", [0, 1])
def test_clamped_kl(agg_mode):
    """grpo_loss_fwd_bwd_kl_clamp: reference log-probs at fixed offsets d from the
    policy's, so that k3(d) lies on both sides of the cap, each value at least
    0.29 from it (the GPU's log-prob error moves k3 by < 0.01)."""
    w = wl.Workload("t", 2, 4, 60, 128, 1500, "uniform", 1, 60, rewards="mix", seed=wl.SEED_BASE + 660)
    c = _case(w, agg_mode)
    kappa, beta = 0.4, 0.5
    rng = np.random.default_rng(w.seed + 9)
    d = rng.choice([-1.5, -0.5, 0.3, 1.0, 1.5], size=w.T)     # k3 = 0.72, 0.11, 0.05, 0.72, 2.98
    ref = (c["want"]["logp"] + d).astype(np.float32)
    args = (c["H"], c["W"], c["y"], c["m"], c["old"], ref, c["adv"], w.n_resp, w.L, w.clip_eps, beta, agg_mode)
    want = oracle.loss_fwd_bwd(*args, kl_clamp=kappa)
    plain = oracle.loss_fwd_bwd(*args)
    capped = ~want["terms"]["kl_inside"] & (c["m"] != 0)
    assert 0.2 < capped.mean() / (c["m"] != 0).mean() < 0.8
    assert rel_fro(want["dW"], plain["dW"]) > 5 * GRAD_RTOL      # the cap changes the gradient visibly
    dd = _dev(c)
    ws = grpo.workspace(w.T, w.Hd, w.V, grpo.GRPO_WS_LOSS, DEV)
    loss, dH, dW = grpo.loss_fwd_bwd(dd["H"], dd["W"], dd["y"], dd["m"], dd["old"], dev_tensor(ref, torch.float32),
                                     dd["adv"], w.n_resp, w.L, w.clip_eps, beta, agg_mode, ws=ws, kl_clamp=kappa)
    assert grpo.check_device_status(ws) == grpo.GRPO_OK
    scale = loss_scale(want["loss"], want["terms"]["w"], want["terms"]["ell"])
    assert abs(loss.item() - want["loss"]) <= LOSS_RTOL * scale, (loss.item(), want["loss"])
    assert rel_fro(dH.double().cpu().numpy(), want["dH"]) <= GRAD_RTOL
    assert rel_fro(dW.double().cpu().numpy(), want["dW"]) <= GRAD_RTOL
    # an infinite cap is the plain entry point, bit for bit
    a = grpo.loss_fwd_bwd(dd["H"], dd["W"], dd["y"], dd["m"], dd["old"], dev_tensor(ref, torch.float32), dd["adv"],
                          w.n_resp, w.L, w.clip_eps, beta, agg_mode, kl_clamp=float("inf"))
    b = grpo.loss_fwd_bwd(dd["H"], dd["W"], dd["y"], dd["m"], dd["old"], dev_tensor(ref, torch.float32), dd["adv"],
                          w.n_resp, w.L, w.clip_eps, beta, agg_mode)
    for x, y in zip(a, b):
        assert torch.equal(x, y)


KEPT_SHAPES = [
    # (n_prompts, G, L, Hd, V, vocabulary chunk or None, tile pair)
    (1, 4, 64, 256, 4096, None, "1"),          # the tiny workload's shape
    (2, 4, 90, 320, 1800, "512", "1"),         # several chunks, a tail chunk of 264 columns
    (3, 4, 60, 192, 1001, "256", "1"),         # odd vocabulary: a tail of 233 columns (not a multiple of 8)
    (3, 4, 60, 192, 2100, "768", "0"),         # 128 x 256 single-CTA tiles
    (2, 3, 200, 128, 777, None, "1"),          # rows past one 256-row tile, one chunk narrower than a tile
]


@pytest.mark.parametrize("agg_mode", [0, 1])
@pytest.mark.parametrize("shape", KEPT_SHAPES)
def test_kept_logits_match_oracle_and_recompute(shape, agg_mode, monkeypatch):
    """A GRPO_WS_LOSS_LOGITS workspace: the forward stores the fp32 logits and
    the backward forms dZ from them.  The results meet the oracle bar and equal
    those of the backward that recomputes the logits, bit for bit."""
    P, G, L, Hd, V, chunk, pair = shape
    if chunk:
        monkeypatch.setenv("GRPO_VOCAB_CHUNK", chunk)
    monkeypatch.setenv("GRPO_CTA_PAIR", pair)
    w = wl.Workload("t", P, G, L, Hd, V, "uniform", 1, L, rewards="mix", seed=wl.SEED_BASE + 5300 + V + Hd)
    c = _case(w, agg_mode)
    kept = _check_fwd_bwd(c, agg_mode, kind=grpo.GRPO_WS_LOSS_LOGITS)
    plain = _check_fwd_bwd(c, agg_mode, kind=grpo.GRPO_WS_LOSS)
    for a, b in zip(kept, plain):
        assert torch.equal(a, b)


def test_kept_logits_lean_workspace_and_capacity(monkeypatch):
    """A kept-logits workspace sized for the unmasked rows works like the plain
    lean one (same bits); a batch with more unmasked rows than it holds reports
    GRPO_ERR_CAPACITY instead of writing past the logits."""
    monkeypatch.setenv("GRPO_VOCAB_CHUNK", "512")
    w = wl.Workload("t", 2, 4, 160, 192, 1500, "uniform", 1, 40, rewards="mix", seed=wl.SEED_BASE + 5400)
    c = _case(w)
    nv = int(c["m"].sum())
    assert nv <= 256 < w.T
    d = _dev(c)
    res = []
    for kind in (grpo.GRPO_WS_LOSS_LOGITS, grpo.GRPO_WS_LOSS):
        ws = grpo.workspace(w.T, w.Hd, w.V, kind, DEV, max_valid=nv)
        assert grpo.loss_plan(w.T, w.Hd, w.V, ws.numel()) == (int(kind == grpo.GRPO_WS_LOSS_LOGITS), 256)
        res.append(grpo.loss_fwd_bwd(d["H"], d["W"], d["y"], d["m"], d["old"], d["ref"], d["adv"],
                                     w.n_resp, w.L, w.clip_eps, w.beta, 0, ws=ws))
        assert grpo.check_device_status(ws) == grpo.GRPO_OK
    for a, b in zip(*res):
        assert torch.equal(a, b)
    assert rel_fro(res[0][2].double().cpu().numpy(), c["want"]["dW"]) <= GRAD_RTOL
    # every row unmasked: 1280 rows against a capacity of 256
    ws = grpo.workspace(w.T, w.Hd, w.V, grpo.GRPO_WS_LOSS_LOGITS, DEV, max_valid=nv)
    grpo.loss_fwd_bwd(d["H"], d["W"], d["y"], torch.ones_like(d["m"]), d["old"], d["ref"], d["adv"], w.n_resp,
                      w.L, w.clip_eps, w.beta, 0, ws=ws)
    assert grpo.check_device_status(ws) == grpo.GRPO_ERR_CAPACITY
    _check_fwd_bwd(c, kind=grpo.GRPO_WS_LOSS_LOGITS)    # a full workspace on the same context


def test_entry_points_agree_across_workspaces(monkeypatch):
    """Every loss entry point (global normaliser, KL cap, per-chunk events,
    dW streamed to pinned host memory, fused AdamW) gives the same bits with a
    kept-logits workspace as with the plain one that recomputes the logits."""
    monkeypatch.setenv("GRPO_VOCAB_CHUNK", "512")
    w = wl.Workload("t", 2, 4, 70, 192, 1700, "uniform", 1, 70, rewards="mix", seed=wl.SEED_BASE + 5500)
    c = _case(w)
    d = _dev(c)
    nv = float(c["m"].sum())
    args = (d["H"], d["W"], d["y"], d["m"], d["old"], d["ref"], d["adv"], w.n_resp, w.L, w.clip_eps, w.beta, 0)
    n_chunks = -(-w.V // grpo.vocab_chunk_cols(w.V))
    assert n_chunks == 4

    def run(kind):
        ws = grpo.workspace(w.T, w.Hd, w.V, kind, DEV)
        out = [grpo.loss_fwd_bwd(*args, ws=ws, norm=2.5 * nv),
               grpo.loss_fwd_bwd(*args, ws=ws, kl_clamp=0.05)]
        events = [torch.cuda.Event() for _ in range(n_chunks)]
        out.append(grpo.loss_fwd_bwd(*args, ws=ws, chunk_events=events))
        host = (torch.empty(1).pin_memory(), torch.empty(w.T, w.Hd).pin_memory(),
                torch.empty(w.V, w.Hd).pin_memory())
        out.append(grpo.loss_fwd_bwd(*args, ws=ws, out=host))
        rng = np.random.default_rng(3)
        master = dev_tensor(oracle.widen_bf16(c["W"]).astype(np.float32), torch.float32)
        ea = torch.zeros_like(master)
        eas = dev_tensor((1e-4 * rng.random(master.shape)).astype(np.float32), torch.float32)
        W_out = torch.empty_like(d["W"])
        lo, dH = grpo.loss_fwd_bwd_adamw(*args[:9], master, ea, eas, 1, lr=1e-3, W_out=W_out, ws=ws)
        out.append((lo, dH, master, ea, eas, W_out))
        torch.cuda.synchronize()
        assert grpo.check_device_status(ws) == grpo.GRPO_OK
        return out

    kept, plain = run(grpo.GRPO_WS_LOSS_LOGITS), run(grpo.GRPO_WS_LOSS)
    for a, b in zip(kept, plain):
        for x, y in zip(a, b):
            assert torch.equal(x.cpu(), y.cpu())
    assert not torch.equal(kept[0][0], kept[1][0])      # the cap and the normaliser change the loss


def test_fwd_bwd_is_deterministic():
    c = _case(wl.Workload("t", 1, 4, 70, 256, 2000, "uniform", 5, 70, seed=wl.SEED_BASE + 600))
    a = _check_fwd_bwd(c)
    b = _check_fwd_bwd(c)
    for x, y in zip(a, b):
        assert torch.equal(x, y)


def test_one_token_per_response_and_zero_std_groups():
    w = wl.Workload("t", 4, 4, 3, 128, 700, "uniform", 1, 1, rewards="bern", zero_std_every=2,
                    seed=wl.SEED_BASE + 700)
    c = _case(w)
    assert c["m"].reshape(w.n_resp, w.L).sum(1).tolist() == [1] * w.n_resp
    _check_fwd_bwd(c)


def test_all_masked_batch():
    w = wl.Workload("t", 1, 2, 40, 64, 500, seed=wl.SEED_BASE + 800)
    c = _case(w)
    d = _dev(c)
    m0 = torch.zeros_like(d["m"])
    loss, dH, dW = grpo.loss_fwd_bwd(d["H"], d["W"], d["y"], m0, d["old"], d["ref"], d["adv"], w.n_resp, w.L)
    assert loss.item() == 0.0 and not dH.any() and not dW.any()
    lp = grpo.token_logprobs(d["H"], d["W"], d["y"], m0)
    assert not lp.any()


def test_bad_target_sets_device_status():
    w = wl.Workload("t", 1, 2, 40, 64, 500, seed=wl.SEED_BASE + 900)
    c = _case(w)
    d = _dev(c)
    y = d["y"].clone()
    y[3] = w.V + 5
    ws = grpo.workspace(w.T, w.Hd, w.V, grpo.GRPO_WS_LOGPROBS, DEV)
    lp = grpo.token_logprobs(d["H"], d["W"], y, d["m"], ws=ws)
    assert grpo.check_device_status(ws) == grpo.GRPO_ERR_DEVICE_CHECK
    assert lp[3].item() == 0.0
    ok = np.flatnonzero(c["m"])
    ok = ok[ok != 3]
    want, _ = oracle.token_logprobs(c["H"], c["W"], c["y"], c["m"])
    assert np.abs(lp.cpu().numpy()[ok] - want[ok]).max() <= LOGP_ATOL
    # the next good call clears the word
    grpo.token_logprobs(d["H"], d["W"], d["y"], d["m"], ws=ws)
    assert grpo.check_device_status(ws) == grpo.GRPO_OK


def test_invalid_group_size_rejected():
    with pytest.raises(grpo.GrpoError) as e:
        grpo.group_advantages(torch.zeros(8, device=DEV), 1)
    assert e.value.status == grpo.GRPO_ERR_INVALID_ARG


# ---------------------------------------------------------------- tile and split boundaries

@pytest.mark.parametrize("n_valid,V", [(1, 100), (255, 256), (256, 4096), (257, 4097), (512, 8191),
                                       (511, 65), (1000, 12288)])
def test_logprobs_at_tile_and_split_boundaries(n_valid, V):
    """Valid-row counts around the 256-row tile, vocabularies around the 256-column tile
    and the 4096-column split, down to a single token and a single partial tile."""
    Hd = 64
    w = wl.Workload("b", 1, 2, (n_valid + 1) // 2 + 3, Hd, V, seed=wl.SEED_BASE + 4000 + n_valid + V)
    Hb, Wb, y = wl.gen_hidden(w), wl.gen_weight(w.with_(w_std=0.3)), wl.gen_targets(w)
    m = np.zeros(w.T, np.uint8)
    m[np.random.default_rng(n_valid).choice(w.T, n_valid, replace=False)] = 1
    want, _ = oracle.token_logprobs(Hb, Wb, y, m)
    got = grpo.token_logprobs(dev_tensor(Hb, torch.bfloat16), dev_tensor(Wb, torch.bfloat16),
                              dev_tensor(y, torch.int32), dev_tensor(m, torch.uint8)).cpu().numpy()
    assert np.all(got[m == 0] == 0.0)
    assert np.abs(got - want).max() <= LOGP_ATOL


@pytest.mark.parametrize("n_valid,V,Hd", [(1, 100, 64), (257, 300, 128), (300, 4097, 64)])
def test_fwd_bwd_at_boundaries(n_valid, V, Hd, monkeypatch):
    monkeypatch.setenv("GRPO_VOCAB_CHUNK", "256")
    G, L = 2, (n_valid + 1) // 2 + 2
    w = wl.Workload("b", 1, G, L, Hd, V, rewards="mix", seed=wl.SEED_BASE + 4500 + n_valid)
    c = _case(w)
    m = np.zeros(w.T, np.uint8)
    m[:n_valid] = 1                                   # response 0 full, response 1 partly (or empty)
    c["m"] = m
    c["want"] = oracle.loss_fwd_bwd(c["H"], c["W"], c["y"], m, c["old"], c["ref"], c["adv"], w.n_resp, w.L,
                                    w.clip_eps, w.beta)
    _check_fwd_bwd(c)


def test_host_output_buffers_stream_dw(monkeypatch):
    """Pinned host outputs: dW arrives chunk by chunk through grpo_loss_fwd_bwd_to_host
    and equals the device-output call bit for bit."""
    monkeypatch.setenv("GRPO_VOCAB_CHUNK", "512")
    c = _case(wl.Workload("t", 2, 4, 48, 128, 1800, "uniform", 1, 48, rewards="mix", seed=wl.SEED_BASE + 660))
    w, d = c["w"], _dev(c)
    dev_out = grpo.loss_fwd_bwd(d["H"], d["W"], d["y"], d["m"], d["old"], d["ref"], d["adv"], w.n_resp, w.L)
    host = (torch.empty(1).pin_memory(), torch.empty(w.T, w.Hd).pin_memory(), torch.empty(w.V, w.Hd).pin_memory())
    got = grpo.loss_fwd_bwd(d["H"], d["W"], d["y"], d["m"], d["old"], d["ref"], d["adv"], w.n_resp, w.L, out=host)
    assert all(g is h for g, h in zip(got, host))
    for g, x in zip(got, dev_out):
        assert torch.equal(g, x.cpu())


def test_larger_hidden_and_vocabulary():
    """Beyond the 8B shape: a 262147-entry vocabulary (65 forward splits, odd tail)
    for the log-probs, and hidden 8192 (128 k-blocks per tile) with a
    40000-entry vocabulary through the whole loss forward + backward."""
    w = wl.Workload("t", 1, 2, 70, 2048, 262147, "uniform", 40, 70, seed=wl.SEED_BASE + 1700)
    Hb, Wb, y, m = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_targets(w), wl.gen_mask(w)
    want, _ = oracle.token_logprobs(Hb, Wb, y, m)
    got = grpo.token_logprobs(dev_tensor(Hb, torch.bfloat16), dev_tensor(Wb, torch.bfloat16),
                              dev_tensor(y, torch.int32), dev_tensor(m, torch.uint8)).cpu().numpy()
    assert np.all(got[m == 0] == 0.0)
    assert np.abs(got.astype(np.float64) - want).max() <= LOGP_ATOL
    w2 = wl.Workload("t", 1, 4, 60, 8192, 40000, "uniform", 20, 60, rewards="mix", seed=wl.SEED_BASE + 1701)
    _check_fwd_bwd(_case(w2))


def test_workspace_sized_for_the_unmasked_rows(monkeypatch):
    """A workspace sized by grpo_workspace_bytes_rows for the batch's unmasked
    rows gives bit-identical log-probs, draws, loss and gradients."""
    monkeypatch.setenv("GRPO_VOCAB_CHUNK", "768")
    w = wl.Workload("t", 4, 4, 200, 128, 2100, "loguniform", 4, 200, rewards="mix", seed=wl.SEED_BASE + 580)
    c = _case(w)
    d = _dev(c)
    nv = int(c["m"].sum())
    assert 256 < nv < w.T - 512          # ragged: the lean workspace is smaller than the full one
    for which in (grpo.GRPO_WS_LOSS, grpo.GRPO_WS_LOGPROBS, grpo.GRPO_WS_SAMPLE):
        assert grpo.workspace_bytes_rows(w.T, nv, w.Hd, w.V, which) < grpo.workspace_bytes(w.T, w.Hd, w.V, which)
    lean = lambda which: grpo.workspace(w.T, w.Hd, w.V, which, DEV, max_valid=nv)
    args = (d["H"], d["W"], d["y"], d["m"], d["old"], d["ref"], d["adv"], w.n_resp, w.L, w.clip_eps, w.beta, 0)
    ws = lean(grpo.GRPO_WS_LOSS)
    a = grpo.loss_fwd_bwd(*args, ws=ws)
    assert grpo.check_device_status(ws) == grpo.GRPO_OK
    b = grpo.loss_fwd_bwd(*args)
    for x, y in zip(a, b):
        assert torch.equal(x, y)
    ws = lean(grpo.GRPO_WS_LOGPROBS)
    assert torch.equal(grpo.token_logprobs(d["H"], d["W"], d["y"], d["m"], ws=ws),
                       grpo.token_logprobs(d["H"], d["W"], d["y"], d["m"]))
    ws = lean(grpo.GRPO_WS_SAMPLE)
    t1, l1 = grpo.sample_tokens(d["H"], d["W"], d["m"], 1.0, seed=5, ws=ws)
    t2, l2 = grpo.sample_tokens(d["H"], d["W"], d["m"], 1.0, seed=5)
    assert torch.equal(t1, t2) and torch.equal(l1, l2)


def test_more_unmasked_rows_than_the_workspace_holds():
    """Past the row capacity the device reports GRPO_ERR_CAPACITY (the count is
    only known there); the rows past it get no output, nothing faults, and the
    next call with a large enough workspace is correct."""
    w = wl.Workload("t", 2, 4, 100, 128, 1500, "uniform", 60, 100, rewards="mix", seed=wl.SEED_BASE + 590)
    c = _case(w)
    d = _dev(c)
    nv = int(c["m"].sum())
    assert nv > 512
    ws = grpo.workspace(w.T, w.Hd, w.V, grpo.GRPO_WS_LOSS, DEV, max_valid=300)   # 512 rows
    grpo.loss_fwd_bwd(d["H"], d["W"], d["y"], d["m"], d["old"], d["ref"], d["adv"], w.n_resp, w.L, w.clip_eps,
                      w.beta, 0, ws=ws)
    assert grpo.check_device_status(ws) == grpo.GRPO_ERR_CAPACITY
    ws_lp = grpo.workspace(w.T, w.Hd, w.V, grpo.GRPO_WS_LOGPROBS, DEV, max_valid=300)
    lp = grpo.token_logprobs(d["H"], d["W"], d["y"], d["m"], ws=ws_lp)
    assert grpo.check_device_status(ws_lp) == grpo.GRPO_ERR_CAPACITY
    idx = wl.valid_index(c["m"])
    assert not lp.cpu().numpy()[idx[512:]].any()       # no output past the capacity
    _check_fwd_bwd(c)                                   # a full workspace on the same context


def test_empty_batches():
    """T = 0: every call accepts it and returns empty outputs (nothing launched
    that reads the inputs); a zero-row noise block is a no-op."""
    Hd, V = 128, 500
    H = torch.empty(0, Hd, dtype=torch.bfloat16, device=DEV)
    W = dev_tensor(wl.gen_weight(wl.Workload("t", 1, 2, 1, Hd, V, seed=wl.SEED_BASE + 1)), torch.bfloat16)
    y = torch.empty(0, dtype=torch.int32, device=DEV)
    m = torch.empty(0, dtype=torch.uint8, device=DEV)
    assert grpo.token_logprobs(H, W, y, m).numel() == 0
    assert grpo.token_logprobs_heads(H, [W, W], y, m).shape == (2, 0)
    tok, lp = grpo.sample_tokens(H, W, m, 1.0, seed=3)
    assert tok.numel() == 0 and lp.numel() == 0
    assert grpo.gumbel_noise(5, 0, V, seed=1).shape == (0, V)
    adv = grpo.group_advantages(torch.empty(0, dtype=torch.float32, device=DEV), 4)
    assert adv.numel() == 0


def test_binding_rejects_mismatched_shapes():
    """The C ABI takes pointers and sizes only; the binding checks every shape,
    output and workspace first, so a mismatch raises instead of reading past a
    buffer."""
    w = wl.Workload("t", 1, 2, 40, 64, 300, "uniform", 1, 40, seed=wl.SEED_BASE + 970)
    c = _case(w)
    d = _dev(c)
    args = [d["H"], d["W"], d["y"], d["m"], d["old"], d["ref"], d["adv"], w.n_resp, w.L]
    bad_cases = [
        (1, d["W"][:, :32]),            # hidden size differs from H
        (2, d["y"][:-1]),               # one target short
        (3, d["m"][:-1]),               # mask short
        (4, d["old"][:-1]),
        (6, d["adv"][:-1]),             # advantages for fewer responses
        (8, w.L + 1),                   # n_resp * L != rows of H
    ]
    for i, v in bad_cases:
        a = list(args)
        a[i] = v
        with pytest.raises(ValueError):
            grpo.loss_fwd_bwd(*a)
    with pytest.raises(ValueError):
        grpo.token_logprobs(d["H"], d["W"], d["y"][:-1], d["m"])
    with pytest.raises(ValueError):
        grpo.loss_fwd_bwd(*args, out=(torch.empty(1, device=DEV), torch.empty(w.T, w.Hd, device=DEV),
                                      torch.empty(w.V - 1, w.Hd, device=DEV)))
    with pytest.raises(ValueError):
        grpo.token_logprobs(d["H"], d["W"], d["y"], d["m"], ws=torch.empty(10, dtype=torch.float32, device=DEV))
    with pytest.raises(ValueError):
        grpo.sample_tokens(d["H"], d["W"], d["m"][:-1])
    # and the well-formed call still works
    grpo.loss_fwd_bwd(*args)


def test_paced_forward_gives_the_same_bits(monkeypatch):
    """The forward and sampling GEMMs pace their persistent grid (a bounded
    wait between tiles, for batches of at least 4096 rows); the pace changes
    only when a CTA issues its copies, so the log-probs, the loss and its
    gradients, and a draw are the same bits with the gate off, at its default
    and at its tightest, and match the oracle."""
    w = wl.Workload("t", 4, 4, 512, 128, 4096, "uniform", 200, 512, seed=wl.SEED_BASE + 1650)
    c = _case(w)
    assert int(c["m"].sum()) >= 4096 and w.T >= 4096
    d = _dev(c)
    for pair in ("1", "0"):  # 2-CTA and single-CTA tiles (the gate counts CTAs either way)
        monkeypatch.setenv("GRPO_CTA_PAIR", pair)
        got = {}
        for gate in ("0", "2", "1", None):
            if gate is None:
                monkeypatch.delenv("GRPO_GATE", raising=False)
            else:
                monkeypatch.setenv("GRPO_GATE", gate)
            lp = grpo.token_logprobs(d["H"], d["W"], d["y"], d["m"])
            loss, dH, dW = _check_fwd_bwd(c)
            tok, tlp = grpo.sample_tokens(d["H"], d["W"], d["m"], 1.0, seed=3, offset=1)
            got[gate] = (lp, loss, dH, dW, tok, tlp)
        for gate in ("2", "1", None):
            for x, y in zip(got[gate], got["0"]):
                assert torch.equal(x, y), (pair, gate)
    monkeypatch.delenv("GRPO_CTA_PAIR")


@pytest.mark.parametrize("case", range(10))
def test_random_shapes_match_oracle(case):
    """Seeded random shapes beyond the hand-picked boundaries: hidden sizes
    64..512 (multiples of 64), vocabularies 1..5000 with any tail, group sizes
    2..6, lengths from one token up, ragged masks with empty responses; the
    log-probs, the loss and both gradients against the oracle."""
    rng = np.random.default_rng(9000 + case)
    Hd = int(rng.integers(1, 9)) * 64
    V = int(rng.integers(1, 5001))
    G = int(rng.integers(2, 7))
    L = int(rng.integers(1, 90))
    lo = int(rng.integers(0, L + 1))
    w = wl.Workload("r", int(rng.integers(1, 4)), G, L, Hd, V, "uniform", lo, L, rewards="mix",
                    seed=wl.SEED_BASE + 9000 + case, w_std=float(rng.choice([0.02, 0.1, 0.3])))
    c = _case(w)
    d = _dev(c)
    want, _ = oracle.token_logprobs(c["H"], c["W"], c["y"], c["m"])
    got = grpo.token_logprobs(d["H"], d["W"], d["y"], d["m"]).cpu().numpy()
    assert np.all(got[c["m"] == 0] == 0.0)
    assert np.abs(got.astype(np.float64) - want).max() <= LOGP_ATOL, (Hd, V, G, L)
    _check_fwd_bwd(c)
