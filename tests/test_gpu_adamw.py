"""The AdamW step fused into the dW GEMM (grpo_loss_fwd_bwd_adamw) against the
float64 oracle's dW followed by the oracle's AdamW step."""
import numpy as np
import pytest

import oracle
import workloads as wl
from tests._util import GRAD_RTOL, clear_of_clip_kink, dev_tensor, rel_fro

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2507_05687_gb300 as grpo  # noqa: E402
from paper_2507_05687_gb300 import build as build_mod  # noqa: E402

build_mod.build()
DEV = torch.device("cuda", 0)
LR, B1, B2, EPS, WD, STEP = 1e-3, 0.9, 0.999, 1e-8, 0.01, 5


def _case(monkeypatch, chunk="768"):
    monkeypatch.setenv("GRPO_VOCAB_CHUNK", chunk)   # several chunks, one ragged
    w = wl.Workload("adam", 2, 4, 80, 192, 2000, "uniform", 1, 80, rewards="mix", seed=wl.SEED_BASE + 777)
    Hb, Wb = wl.gen_hidden(w), wl.gen_weight(w)
    y, m, r = wl.gen_targets(w), wl.gen_mask(w), wl.gen_rewards(w)
    old = oracle.token_logprobs(Hb, wl.gen_weight(w, "old", Wb), y, m)[0].astype(np.float32)
    old = clear_of_clip_kink(oracle.token_logprobs(Hb, Wb, y, m)[0], old, w.clip_eps)
    ref = oracle.token_logprobs(Hb, wl.gen_weight(w, "ref", Wb), y, m)[0].astype(np.float32)
    adv = oracle.group_advantages(r, w.G, float(np.float32(w.adv_eps)))
    want = oracle.loss_fwd_bwd(Hb, Wb, y, m, old, ref, adv, w.n_resp, w.L, w.clip_eps, w.beta)
    rng = np.random.default_rng(5)
    theta0 = oracle.widen_bf16(Wb).astype(np.float32)
    m0 = np.zeros_like(theta0)  # first moment from zero: m = (1 - beta1) g exactly
    scale = 10 * np.abs(want["dW"]).mean()
    v0 = (scale * (0.5 + rng.random(theta0.shape))).astype(np.float32) ** 2  # dominant: update linear in g
    return w, Hb, Wb, y, m, old, ref, adv, want, theta0, m0, v0


def _run(w, Hb, Wb, y, m, old, ref, adv, theta0, m0, v0, in_place, ws=None):
    W = dev_tensor(Wb, torch.bfloat16)
    master, ea, eas = (torch.from_numpy(x.copy()).to(DEV) for x in (theta0, m0, v0))
    W_out = W if in_place else torch.empty_like(W)
    loss, dH = grpo.loss_fwd_bwd_adamw(dev_tensor(Hb, torch.bfloat16), W, dev_tensor(y, torch.int32),
                                       dev_tensor(m, torch.uint8), dev_tensor(old, torch.float32),
                                       dev_tensor(ref, torch.float32), dev_tensor(adv, torch.float32), w.n_resp,
                                       w.L, master, ea, eas, STEP, lr=LR, betas=(B1, B2), eps=EPS,
                                       weight_decay=WD, W_out=W_out, ws=ws)
    torch.cuda.synchronize()
    return loss, dH, master, ea, eas, W_out


@pytest.mark.parametrize("pair", ["1", "0"])
def test_fused_adamw_matches_oracle(pair, monkeypatch):
    """Both tile shapes (their operand rings differ: 5 stages of the pair tile,
    3 of the single-CTA tile, to make room for the weight / moment blocks)."""
    monkeypatch.setenv("GRPO_CTA_PAIR", pair)
    w, Hb, Wb, y, m, old, ref, adv, want, theta0, m0, v0 = _case(monkeypatch)
    loss, dH, master, ea, eas, W_out = _run(w, Hb, Wb, y, m, old, ref, adv, theta0, m0, v0, in_place=False)
    th_o, m_o, v_o = oracle.adamw_step(theta0, m0, v0, want["dW"], LR, B1, B2, EPS, WD, STEP)
    g_gpu = ea.double().cpu().numpy() / (1 - B1)                 # the dW the step consumed
    assert rel_fro(g_gpu, want["dW"]) <= GRAD_RTOL
    v_gpu = eas.double().cpu().numpy()
    assert rel_fro(v_gpu - B2 * v0, v_o - B2 * v0) <= 2 * GRAD_RTOL   # (1 - beta2) g^2
    th_gpu = master.double().cpu().numpy()
    assert rel_fro(th_gpu - theta0, th_o - theta0) <= GRAD_RTOL       # the update itself
    # the bf16 weights are the rounded fp32 master weights
    expect_bits = wl.f32_to_bf16_bits(master.cpu().numpy())
    assert np.array_equal(W_out.cpu().view(torch.int16).numpy().view(np.uint16), expect_bits)
    # loss and dH are those of the plain call, bit for bit
    l2, dH2, _ = grpo.loss_fwd_bwd(dev_tensor(Hb, torch.bfloat16), dev_tensor(Wb, torch.bfloat16),
                                   dev_tensor(y, torch.int32), dev_tensor(m, torch.uint8),
                                   dev_tensor(old, torch.float32), dev_tensor(ref, torch.float32),
                                   dev_tensor(adv, torch.float32), w.n_resp, w.L, w.clip_eps, w.beta)
    assert torch.equal(loss, l2) and torch.equal(dH, dH2)


def test_fused_adamw_in_place_weights(monkeypatch):
    """W_out = W: each vocabulary chunk's rows are updated after their last read."""
    args = _case(monkeypatch)
    w, Hb, Wb, y, m, old, ref, adv, want, theta0, m0, v0 = args
    a = _run(w, Hb, Wb, y, m, old, ref, adv, theta0, m0, v0, in_place=False)
    b = _run(w, Hb, Wb, y, m, old, ref, adv, theta0, m0, v0, in_place=True)
    for x, z in zip(a, b):
        assert torch.equal(x, z)


def test_fused_adamw_rejects_bad_hyperparameters():
    w = wl.Workload("adam", 1, 2, 8, 64, 300, seed=wl.SEED_BASE + 778)
    W = torch.zeros(w.V, w.Hd, dtype=torch.bfloat16, device=DEV)
    st = [torch.zeros(w.V, w.Hd, device=DEV) for _ in range(3)]
    z = torch.zeros(w.T, device=DEV)
    for kw in ({"step": 0}, {"betas": (1.0, 0.999)}, {"eps": 0.0}):
        step = kw.pop("step", 1)
        with pytest.raises(grpo.GrpoError) as e:
            grpo.loss_fwd_bwd_adamw(torch.zeros(w.T, w.Hd, dtype=torch.bfloat16, device=DEV), W,
                                    torch.zeros(w.T, dtype=torch.int32, device=DEV),
                                    torch.ones(w.T, dtype=torch.uint8, device=DEV), z, z,
                                    torch.zeros(w.n_resp, device=DEV), w.n_resp, w.L, *st, step, **kw)
        assert e.value.status == grpo.GRPO_ERR_INVALID_ARG


def test_standalone_adamw_matches_oracle():
    rng = np.random.default_rng(11)
    n = 4 * 12345
    th, m0, g = (rng.normal(size=n).astype(np.float32) for _ in range(3))
    v0 = (rng.random(n) * 2).astype(np.float32)
    t = [torch.from_numpy(x.copy()).to(DEV) for x in (th, m0, v0, g)]
    w_out = torch.empty(n, dtype=torch.bfloat16, device=DEV)
    grpo.adamw_step(t[0], t[1], t[2], t[3], w_out, step=3, lr=1e-2, betas=(0.9, 0.99), eps=1e-6, weight_decay=0.1)
    th_o, m_o, v_o = oracle.adamw_step(th, m0, v0, g, 1e-2, 0.9, 0.99, 1e-6, 0.1, 3)
    np.testing.assert_allclose(t[1].cpu().numpy(), m_o, rtol=2e-6, atol=1e-7)
    np.testing.assert_allclose(t[2].cpu().numpy(), v_o, rtol=2e-6, atol=1e-7)
    np.testing.assert_allclose(t[0].cpu().numpy(), th_o, rtol=2e-6, atol=1e-6)
    assert np.array_equal(w_out.cpu().view(torch.int16).numpy().view(np.uint16),
                          wl.f32_to_bf16_bits(t[0].cpu().numpy()))


def test_fused_equals_stored_dw_plus_separate_step(monkeypatch):
    w, Hb, Wb, y, m, old, ref, adv, want, theta0, m0, v0 = _case(monkeypatch)
    _, _, master_f, ea_f, eas_f, wout_f = _run(w, Hb, Wb, y, m, old, ref, adv, theta0, m0, v0, in_place=False)
    _, _, dW = grpo.loss_fwd_bwd(dev_tensor(Hb, torch.bfloat16), dev_tensor(Wb, torch.bfloat16),
                                 dev_tensor(y, torch.int32), dev_tensor(m, torch.uint8),
                                 dev_tensor(old, torch.float32), dev_tensor(ref, torch.float32),
                                 dev_tensor(adv, torch.float32), w.n_resp, w.L, w.clip_eps, w.beta)
    master, ea, eas = (torch.from_numpy(x.copy()).to(DEV) for x in (theta0, m0, v0))
    wout = torch.empty(w.V, w.Hd, dtype=torch.bfloat16, device=DEV)
    grpo.adamw_step(master, ea, eas, dW, wout, STEP, lr=LR, betas=(B1, B2), eps=EPS, weight_decay=WD)
    for a, b in ((master_f, master), (ea_f, ea), (eas_f, eas)):
        torch.testing.assert_close(a, b, rtol=1e-6, atol=1e-9)


@pytest.mark.parametrize("pair", ["1", "0"])
def test_weight_block_wait_that_runs_out_reports_timeout(pair, monkeypatch):
    """Failure detection of the fused step's own wait, without a fault: a test
    hook (GRPO_TEST_DROP_ADAM) makes CTA 0 skip the loads of one weight block,
    the bounded wait for them gives up (0.2 s), the call reports
    GRPO_ERR_TIMEOUT, and the next call on the same context is correct."""
    monkeypatch.setenv("GRPO_CTA_PAIR", pair)
    w, Hb, Wb, y, m, old, ref, adv, want, theta0, m0, v0 = _case(monkeypatch)
    ws = grpo.workspace(w.T, w.Hd, w.V, grpo.GRPO_WS_LOSS, DEV)
    monkeypatch.setenv("GRPO_TEST_DROP_ADAM", "2")
    _run(w, Hb, Wb, y, m, old, ref, adv, theta0, m0, v0, in_place=False, ws=ws)
    assert grpo.check_device_status(ws) == grpo.GRPO_ERR_TIMEOUT
    monkeypatch.delenv("GRPO_TEST_DROP_ADAM")
    loss, dH, master, ea, eas, W_out = _run(w, Hb, Wb, y, m, old, ref, adv, theta0, m0, v0, in_place=False, ws=ws)
    assert grpo.check_device_status(ws) == grpo.GRPO_OK
    th_o, _, _ = oracle.adamw_step(theta0, m0, v0, want["dW"], LR, B1, B2, EPS, WD, STEP)
    assert rel_fro(master.double().cpu().numpy() - theta0, th_o - theta0) <= GRAD_RTOL
