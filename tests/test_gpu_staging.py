"""BatchStager (paper_2507_05687_gb300/staging.py): batches copied from pinned
host memory on a copy stream while the previous step computes.  Each staged
step must see exactly its own batch: with three different batches cycling
through two slots, every step's log-probs and loss equal those of the same
call on a direct device copy, bit for bit, and the slots are refilled only
after the step that read them."""
import numpy as np
import pytest

import workloads as wl
from tests._util import dev_tensor

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2507_05687_gb300 as grpo  # noqa: E402
from paper_2507_05687_gb300 import build as build_mod  # noqa: E402
from paper_2507_05687_gb300.staging import BatchStager  # noqa: E402

build_mod.build()
DEV = torch.device("cuda", 0)


def _batch(seed):
    w = wl.Workload("s", 2, 4, 64, 128, 3000, "uniform", 8, 64, seed=wl.SEED_BASE + seed, w_std=0.05)
    Hb, y, m, r = wl.gen_hidden(w), wl.gen_targets(w), wl.gen_mask(w), wl.gen_rewards(w)
    rng = np.random.default_rng(seed)
    old = (rng.standard_normal(w.T) * 0.01 - 8.0).astype(np.float32)
    ref = (rng.standard_normal(w.T) * 0.01 - 8.0).astype(np.float32)

    def pin(a, dt):
        return torch.from_numpy(np.ascontiguousarray(a)).view(dt).pin_memory()

    host = (pin(Hb, torch.bfloat16), pin(y, torch.int32), pin(m, torch.uint8), pin(old, torch.float32),
            pin(ref, torch.float32), pin(r, torch.float32))
    return w, host


def _step(w, W, H, y, m, old, ref, r, ws):
    adv = grpo.group_advantages(r, w.G, w.adv_eps)
    lp = grpo.token_logprobs(H, W, y, m)
    loss, dH, dW = grpo.loss_fwd_bwd(H, W, y, m, old, ref, adv, w.n_resp, w.L, w.clip_eps, w.beta, ws=ws)
    return lp, loss, dH, dW


def test_staged_batches_match_direct_calls():
    batches = [_batch(s) for s in (5100, 5101, 5102)]
    w = batches[0][0]
    W = dev_tensor(wl.gen_weight(w), torch.bfloat16)
    ws = grpo.loss_workspace(w.T, w.Hd, w.V, DEV)
    want = [[x.clone() for x in _step(w, W, *[t.to(DEV) for t in host], ws)] for w, host in batches]
    stager = BatchStager(DEV)
    order = [0, 1, 2, 0, 2, 1, 1]
    stager.submit(batches[order[0]][1])
    for i, b in enumerate(order):
        dev_batch = stager.get()
        if i + 1 < len(order):
            stager.submit(batches[order[i + 1]][1])
        got = _step(w, W, *dev_batch, ws)
        stager.release()
        for x, y in zip(got, want[b]):
            assert torch.equal(x, y), (i, b)


def test_stager_argument_checks():
    w, host = _batch(5103)
    stager = BatchStager(DEV)
    with pytest.raises(RuntimeError):
        stager.get()
    stager.submit(host)
    stager.submit(host)
    with pytest.raises(RuntimeError):  # both slots hold batches not yet taken
        stager.submit(host)
    with pytest.raises(ValueError):
        BatchStager(DEV, slots=1)
    with pytest.raises(RuntimeError):  # nothing handed out yet
        stager.release()
    stager.get()
    with pytest.raises(RuntimeError):  # the previous batch is not released
        stager.get()
    with pytest.raises(ValueError):
        stager.submit([host[0].to(DEV)])
    with pytest.raises(RuntimeError):  # the next slot (the one handed out) is still in use
        stager.submit(host)
    stager.release()
    stager.get()
    stager.release()
    stager.submit(host)
