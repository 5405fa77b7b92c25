"""The calls capture into CUDA graphs: they allocate nothing, never synchronise
the stream and enqueue only kernels and a memset, so a training step or a
decode step can be replayed as one graph launch.  A replay must equal the eager
call bit for bit (the kernels are deterministic)."""
import numpy as np
import pytest

import oracle
import workloads as wl
from tests._util import clear_of_clip_kink, dev_tensor

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2507_05687_gb300 as grpo  # noqa: E402
from paper_2507_05687_gb300 import build as build_mod  # noqa: E402

build_mod.build()
DEV = torch.device("cuda", 0)


@pytest.mark.parametrize("kind", ["plain", "kept_logits"])
def test_loss_step_replays_from_a_graph(kind, monkeypatch):
    monkeypatch.setenv("GRPO_VOCAB_CHUNK", "768")
    w = wl.Workload("g", 2, 4, 60, 128, 2100, "uniform", 1, 60, rewards="mix", seed=wl.SEED_BASE + 950)
    Hb, Wb, y, m, r = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_targets(w), wl.gen_mask(w), wl.gen_rewards(w)
    lp = oracle.token_logprobs(Hb, Wb, y, m)[0]
    old = clear_of_clip_kink(lp, oracle.token_logprobs(Hb, wl.gen_weight(w, "old", Wb), y, m)[0].astype(np.float32),
                             w.clip_eps)
    ref = oracle.token_logprobs(Hb, wl.gen_weight(w, "ref", Wb), y, m)[0].astype(np.float32)
    H, W = dev_tensor(Hb, torch.bfloat16), dev_tensor(Wb, torch.bfloat16)
    yd, md = dev_tensor(y, torch.int32), dev_tensor(m, torch.uint8)
    oldd, refd, rd = dev_tensor(old, torch.float32), dev_tensor(ref, torch.float32), dev_tensor(r, torch.float32)
    ws = grpo.workspace(w.T, w.Hd, w.V, grpo.GRPO_WS_LOSS if kind == "plain" else grpo.GRPO_WS_LOSS_LOGITS, DEV)
    assert grpo.loss_plan(w.T, w.Hd, w.V, ws.numel())[0] == (kind == "kept_logits")
    adv = torch.empty(w.n_resp, dtype=torch.float32, device=DEV)
    out = (torch.empty(1, device=DEV), torch.empty(w.T, w.Hd, device=DEV), torch.empty(w.V, w.Hd, device=DEV))

    def step():
        grpo.group_advantages(rd, w.G, w.adv_eps, out=adv)
        grpo.loss_fwd_bwd(H, W, yd, md, oldd, refd, adv, w.n_resp, w.L, w.clip_eps, w.beta, 0, ws=ws, out=out)

    side = torch.cuda.Stream(DEV)
    side.wait_stream(torch.cuda.current_stream(DEV))
    with torch.cuda.stream(side):   # warm-up (first-use set-up) outside the capture
        step()
    torch.cuda.current_stream(DEV).wait_stream(side)
    eager = [t.clone() for t in out]
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        step()
    for _ in range(2):
        for t in out:
            t.fill_(float("nan"))
        g.replay()
        torch.cuda.synchronize()
        assert grpo.check_device_status(ws) == grpo.GRPO_OK
        for a, b in zip(out, eager):
            assert torch.equal(a, b)


@pytest.mark.parametrize("top_p", [None, 0.9])
def test_decode_step_draw_replays_from_a_graph(top_p):
    """A decode-step draw, plain or nucleus (its list of rows whose winner falls
    outside is rebuilt on the device every replay), captured and replayed."""
    w = wl.DECODE_WORKLOADS["decode256_8b"].with_(V=32768)
    Hb, Wb, m = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_mask(w)
    H, W, md = dev_tensor(Hb, torch.bfloat16), dev_tensor(Wb, torch.bfloat16), dev_tensor(m, torch.uint8)
    ws = grpo.workspace(w.T, w.Hd, w.V, grpo.GRPO_WS_SAMPLE if top_p is None else grpo.GRPO_WS_SAMPLE_TOP_P, DEV)
    out = (torch.empty(w.T, dtype=torch.int32, device=DEV), torch.empty(w.T, device=DEV))

    def draw():
        if top_p is None:
            return grpo.sample_tokens(H, W, md, 1.0, seed=11, offset=3, ws=ws, out=out)
        return grpo.sample_tokens_top_p(H, W, md, 1.0, top_p, seed=11, offset=3, ws=ws, out=out)

    eager = [t.clone() for t in draw()]
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        draw()
    for _ in range(2):
        out[0].fill_(-7)
        out[1].fill_(float("nan"))
        g.replay()
        torch.cuda.synchronize()
        assert grpo.check_device_status(ws) == grpo.GRPO_OK
        assert torch.equal(out[0], eager[0]) and torch.equal(out[1], eager[1])


def test_calls_on_two_streams_with_their_own_workspaces():
    """Two loss calls in flight at once on different streams (each with its own
    workspace) give what they give one after the other: the library's shared
    state (device properties, tensor-map encoder) is read-only after set-up and
    its kernels never wait on one another across launches."""
    cases = []
    for seed in (960, 961):
        w = wl.Workload("s", 2, 4, 50, 128, 1700, "uniform", 1, 50, rewards="mix", seed=wl.SEED_BASE + seed)
        Hb, Wb, y, m, r = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_targets(w), wl.gen_mask(w), wl.gen_rewards(w)
        lp = oracle.token_logprobs(Hb, Wb, y, m)[0]
        d = [dev_tensor(Hb, torch.bfloat16), dev_tensor(Wb, torch.bfloat16), dev_tensor(y, torch.int32),
             dev_tensor(m, torch.uint8), dev_tensor((lp - 0.05).astype(np.float32), torch.float32),
             dev_tensor((lp + 0.1).astype(np.float32), torch.float32),
             dev_tensor(oracle.group_advantages(r, w.G, float(np.float32(w.adv_eps))), torch.float32)]
        cases.append((w, d))
    seq = [grpo.loss_fwd_bwd(*d, w.n_resp, w.L, w.clip_eps, w.beta, 0) for w, d in cases]
    torch.cuda.synchronize()
    streams = [torch.cuda.Stream(DEV) for _ in cases]
    outs = []
    for (w, d), st in zip(cases, streams):
        st.wait_stream(torch.cuda.current_stream(DEV))
        with torch.cuda.stream(st):
            ws = grpo.workspace(w.T, w.Hd, w.V, grpo.GRPO_WS_LOSS, DEV)
            outs.append(grpo.loss_fwd_bwd(*d, w.n_resp, w.L, w.clip_eps, w.beta, 0, ws=ws))
    torch.cuda.synchronize()
    for a, b in zip(outs, seq):
        for x, y in zip(a, b):
            assert torch.equal(x, y)
