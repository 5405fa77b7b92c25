"""Per-chunk completion events of the loss backward (grpo_loss_fwd_bwd_events)
and the data-parallel call that overlaps each chunk's dW all-reduce with the
later chunks (paper_2507_05687_gb300.dp).

With one GPU, the collective runs in a one-rank NCCL group: the
events, the communication stream and the NCCL calls are the real ones, and a
one-rank sum must leave every bit of loss and dW unchanged.  The sharding and
the global normaliser are covered by the two-rank gloo tests.
"""
import socket

import numpy as np
import pytest

import oracle
import workloads as wl
from tests._util import dev_tensor

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2507_05687_gb300 as grpo  # noqa: E402
from paper_2507_05687_gb300 import build as build_mod, dp  # noqa: E402

build_mod.build()
DEV = torch.device("cuda", 0)


def _inputs(seed):
    w = wl.Workload("t", 2, 4, 70, 128, 2100, "uniform", 1, 70, rewards="mix", seed=wl.SEED_BASE + seed)
    Hb, Wb, y, m, r = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_targets(w), wl.gen_mask(w), wl.gen_rewards(w)
    old = oracle.token_logprobs(Hb, wl.gen_weight(w, "old", Wb), y, m)[0].astype(np.float32)
    ref = oracle.token_logprobs(Hb, wl.gen_weight(w, "ref", Wb), y, m)[0].astype(np.float32)
    adv = oracle.group_advantages(r, w.G, float(np.float32(w.adv_eps)))
    d = dict(H=dev_tensor(Hb, torch.bfloat16), W=dev_tensor(Wb, torch.bfloat16), y=dev_tensor(y, torch.int32),
             m=dev_tensor(m, torch.uint8), old=dev_tensor(old, torch.float32), ref=dev_tensor(ref, torch.float32),
             adv=dev_tensor(adv, torch.float32))
    return w, d, int(m.sum())


def test_chunk_events_fire_after_their_rows(monkeypatch):
    """A side stream that waits on event c and snapshots chunk c's rows of dW
    (prefilled with NaN) must see the final values of those rows."""
    monkeypatch.setenv("GRPO_VOCAB_CHUNK", "768")
    w, d, nv = _inputs(900)
    rows = dp.chunk_rows(w.V, grpo.vocab_chunk_cols(w.V))
    assert len(rows) == 3
    out = (torch.empty(1, device=DEV), torch.empty(w.T, w.Hd, device=DEV),
           torch.full((w.V, w.Hd), float("nan"), device=DEV))
    events = [torch.cuda.Event() for _ in rows]
    side = torch.cuda.Stream(DEV)
    snaps = [torch.empty(r.stop - r.start, w.Hd, device=DEV) for r in rows]
    loss, dH, dW = grpo.loss_fwd_bwd(d["H"], d["W"], d["y"], d["m"], d["old"], d["ref"], d["adv"], w.n_resp, w.L,
                                     w.clip_eps, w.beta, 0, out=out, chunk_events=events)
    with torch.cuda.stream(side):
        for ev, r, sn in zip(events, rows, snaps):
            side.wait_event(ev)
            sn.copy_(dW[r])
    torch.cuda.synchronize()
    for r, sn in zip(rows, snaps):
        assert torch.equal(sn, dW[r])
    plain = grpo.loss_fwd_bwd(d["H"], d["W"], d["y"], d["m"], d["old"], d["ref"], d["adv"], w.n_resp, w.L,
                              w.clip_eps, w.beta, 0)
    for a, b in zip((loss, dH, dW), plain):
        assert torch.equal(a, b)
    with pytest.raises(grpo.GrpoError):
        grpo.loss_fwd_bwd(d["H"], d["W"], d["y"], d["m"], d["old"], d["ref"], d["adv"], w.n_resp, w.L,
                          w.clip_eps, w.beta, 0, chunk_events=events[:2])


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_overlapped_allreduce_one_rank_nccl(monkeypatch):
    import torch.distributed as dist
    monkeypatch.setenv("GRPO_VOCAB_CHUNK", "512")
    monkeypatch.setenv("NCCL_NVLS_ENABLE", "0")
    w, d, nv = _inputs(901)
    dist.init_process_group("nccl", init_method=f"tcp://127.0.0.1:{_free_port()}", rank=0, world_size=1,
                            device_id=DEV)
    try:
        loss, dH, dW = dp.dp_loss_fwd_bwd(d["H"], d["W"], d["y"], d["m"], d["old"], d["ref"], d["adv"], w.n_resp,
                                          w.L, w.clip_eps, w.beta, 0, float(nv))
        torch.cuda.synchronize()
    finally:
        dist.destroy_process_group()
    want = grpo.loss_fwd_bwd(d["H"], d["W"], d["y"], d["m"], d["old"], d["ref"], d["adv"], w.n_resp, w.L,
                             w.clip_eps, w.beta, 0, norm=float(nv))
    for a, b in zip((loss, dH, dW), want):
        assert torch.equal(a, b)
