"""The workspace-free log-prob entry point, grpo_token_logprobs_noalloc.

Some callers cannot hand the library a workspace: they run where cudaMalloc
is forbidden or would stall the whole device (inside a CUDA stream capture,
in a latency-critical loop that must not allocate after start-up), or they
reach the library from a language binding that has no device allocator.  For
them the library keeps a fixed 64 MiB scratch array in its own device memory.

This file checks, through the C ABI, that the workspace-free call gives the
same log-probs as grpo_token_logprobs with a caller workspace, bit for bit
(the same kernels on the same inputs), and the float64 oracle's within the
log-prob tolerance, on two calls in a row of different sizes, so that state
the first call leaves in the shared array cannot leak into the second; that a
bad target in a no-alloc call is reported by grpo_noalloc_check_status and
cleared by the next call; and that sizes beyond the array are refused.  It is
named so pytest collects it last.
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
STATIC_BYTES = 64 << 20


def _host(w):
    return wl.gen_hidden(w), wl.gen_weight(w), wl.gen_targets(w), wl.gen_mask(w)


def _noalloc(H, W, y, m):
    lib = grpo.load()
    T, Hd = H.shape
    V = W.shape[0]
    out = torch.full((T,), float("nan"), dtype=torch.float32, device=DEV)
    st = lib.grpo_token_logprobs_noalloc(H.data_ptr(), W.data_ptr(), y.data_ptr(), m.data_ptr(), T, Hd, V,
                                         out.data_ptr(), torch.cuda.current_stream(DEV).cuda_stream)
    assert st == grpo.GRPO_OK, grpo.status_string(st)
    return out


def _status():
    return grpo.load().grpo_noalloc_check_status(torch.cuda.current_stream(DEV).cuda_stream)


CASES = [
    # a larger batch first, then a smaller one with a vocabulary tail, so the
    # second call runs on an array holding the first call's leftovers
    wl.Workload("na1", 2, 4, 300, 512, 9000, "uniform", 1, 300, seed=wl.SEED_BASE + 4242),
    wl.Workload("na2", 1, 3, 77, 256, 1000, "uniform", 1, 77, seed=wl.SEED_BASE + 4343),
]


def test_noalloc_matches_workspace_call_and_oracle_twice_in_a_row():
    for w in CASES:
        assert grpo.workspace_bytes(w.T, w.Hd, w.V, grpo.GRPO_WS_LOGPROBS) <= STATIC_BYTES
        Hb, Wb, yb, mb = _host(w)
        H, W = dev_tensor(Hb, torch.bfloat16), dev_tensor(Wb, torch.bfloat16)
        y, m = dev_tensor(yb, torch.int32), dev_tensor(mb, torch.uint8)
        want = grpo.token_logprobs(H, W, y, m)
        got = _noalloc(H, W, y, m)
        assert _status() == grpo.GRPO_OK
        g, e = got.cpu().numpy(), want.cpu().numpy()
        assert np.array_equal(g.view(np.uint32), e.view(np.uint32))
        assert np.all(g[mb == 0] == 0.0)
        ref, _ = oracle.token_logprobs(Hb, Wb, yb, mb)
        assert np.abs(g.astype(np.float64) - ref).max() <= LOGP_ATOL


def test_noalloc_reports_a_bad_target_and_clears_it():
    w = CASES[1]
    Hb, Wb, yb, mb = _host(w)
    bad = yb.copy()
    t_bad = int(wl.valid_index(mb)[3])
    bad[t_bad] = w.V + 5    # outside [0, V) on an unmasked row
    H, W = dev_tensor(Hb, torch.bfloat16), dev_tensor(Wb, torch.bfloat16)
    m = dev_tensor(mb, torch.uint8)
    got = _noalloc(H, W, dev_tensor(bad, torch.int32), m).cpu().numpy()
    assert _status() == grpo.GRPO_ERR_DEVICE_CHECK
    assert got[t_bad] == 0.0
    # the other rows are those of a good call
    ref, _ = oracle.token_logprobs(Hb, Wb, yb, mb)
    keep = np.ones(w.T, bool)
    keep[t_bad] = False
    assert np.abs(got[keep].astype(np.float64) - ref[keep]).max() <= LOGP_ATOL
    # the next call starts with a clear word
    _noalloc(H, W, dev_tensor(yb, torch.int32), m)
    assert _status() == grpo.GRPO_OK


def test_noalloc_refuses_sizes_beyond_its_array():
    lib = grpo.load()
    Hd, V = 4096, 155136
    T = 7681  # one token more than 64 MiB of scratch holds at this shape
    assert grpo.workspace_bytes(T, Hd, V, grpo.GRPO_WS_LOGPROBS) > STATIC_BYTES
    fake = 0x10000  # never dereferenced: the size check comes first
    st = lib.grpo_token_logprobs_noalloc(fake, fake, fake, fake, T, Hd, V, fake, None)
    assert st == grpo.GRPO_ERR_WORKSPACE
    assert lib.grpo_token_logprobs_noalloc(fake, fake, fake, fake, 10, 60, V, fake, None) == grpo.GRPO_ERR_INVALID_ARG
