"""Failure detection on the GPU without a fault: a pipeline wait that runs out.

A test hook (GRPO_TEST_DROP_KBLOCK) makes CTA 0 of the forward GEMM skip the
copies of one k-block, so the MMA issuer's wait for that stage never
completes.  The bounded wait (0.2 s under the hook) gives up, every role of the
CTA (pair) unwinds, TMEM is released, and the device status word reports
GRPO_ERR_TIMEOUT.  The context stays usable: the next call is correct.
"""
import numpy as np
import pytest

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


@pytest.mark.parametrize("pair", ["1", "0"])
def test_wait_that_runs_out_reports_timeout_and_context_survives(pair, monkeypatch):
    monkeypatch.setenv("GRPO_CTA_PAIR", pair)
    w = wl.Workload("f", 2, 4, 200, 256, 3000, "uniform", 20, 200, seed=wl.SEED_BASE + 3100)
    Hb, Wb, y, m = wl.gen_hidden(w), wl.gen_weight(w), wl.gen_targets(w), wl.gen_mask(w)
    H, W = dev_tensor(Hb, torch.bfloat16), dev_tensor(Wb, torch.bfloat16)
    yd, md = dev_tensor(y, torch.int32), dev_tensor(m, torch.uint8)
    ws = grpo.workspace(w.T, w.Hd, w.V, grpo.GRPO_WS_LOGPROBS, DEV)

    monkeypatch.setenv("GRPO_TEST_DROP_KBLOCK", "3")
    grpo.token_logprobs(H, W, yd, md, ws=ws)              # enqueues fine; the device gives up
    assert grpo.check_device_status(ws) == grpo.GRPO_ERR_TIMEOUT

    monkeypatch.delenv("GRPO_TEST_DROP_KBLOCK")
    lp = grpo.token_logprobs(H, W, yd, md, ws=ws)         # same context, same workspace
    assert grpo.check_device_status(ws) == grpo.GRPO_OK
    want, _ = oracle.token_logprobs(Hb, Wb, y, m)
    assert np.abs(lp.cpu().numpy() - want).max() <= LOGP_ATOL
