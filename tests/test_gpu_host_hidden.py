"""Hidden states left in page-locked host memory (include/grpo.h: H may be
registered host memory; the row gather reads the unmasked rows over the host
link).  The results are the same bits as with H on the device, for the
log-prob, scoring, sampling and loss calls, and through the C ABI pageable
host memory is refused with GRPO_ERR_INVALID_ARG before anything runs."""
import ctypes

import numpy as np
import pytest

import workloads as wl
from tests._util import dev_tensor

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2507_05687_gb300 as grpo  # noqa: E402
from paper_2507_05687_gb300 import binding  # noqa: E402
from paper_2507_05687_gb300 import build as build_mod  # noqa: E402

build_mod.build()
DEV = torch.device("cuda", 0)

W_SMALL = wl.Workload("h", 3, 4, 70, 192, 5000, "uniform", 20, 70, seed=wl.SEED_BASE + 3400, w_std=0.05)


def _inputs(w):
    Hb, Wb = wl.gen_hidden(w), wl.gen_weight(w)
    y, m, r = wl.gen_targets(w), wl.gen_mask(w), wl.gen_rewards(w)
    Hp = torch.from_numpy(np.ascontiguousarray(Hb)).view(torch.bfloat16).pin_memory()
    return Hb, Wb, y, m, r, Hp


def test_host_hidden_states_give_the_same_bits():
    w = W_SMALL
    Hb, Wb, y, m, r, Hp = _inputs(w)
    assert Hp.is_pinned()
    Hd, Wd = dev_tensor(Hb, torch.bfloat16), dev_tensor(Wb, torch.bfloat16)
    yd, md = dev_tensor(y, torch.int32), dev_tensor(m, torch.uint8)
    a = grpo.token_logprobs(Hd, Wd, yd, md)
    b = grpo.token_logprobs(Hp, Wd, yd, md)
    assert b.is_cuda and torch.equal(a, b)
    W2 = dev_tensor(wl.gen_weight(w, "old", Wb), torch.bfloat16)
    assert torch.equal(grpo.token_logprobs_heads(Hd, [Wd, W2], yd, md), grpo.token_logprobs_heads(Hp, [Wd, W2], yd, md))
    ta, la = grpo.sample_tokens(Hd, Wd, md, 1.0, seed=5, offset=2)
    tb, lb = grpo.sample_tokens(Hp, Wd, md, 1.0, seed=5, offset=2)
    assert torch.equal(ta, tb) and torch.equal(la, lb)
    ta, la = grpo.sample_tokens_top_p(Hd, Wd, md, 1.0, 0.8, seed=5, offset=2)
    tb, lb = grpo.sample_tokens_top_p(Hp, Wd, md, 1.0, 0.8, seed=5, offset=2)
    assert torch.equal(ta, tb) and torch.equal(la, lb)
    adv = grpo.group_advantages(dev_tensor(r, torch.float32), w.G, w.adv_eps)
    old = a.clone()
    ref = (a - 0.01).contiguous()
    la, dHa, dWa = grpo.loss_fwd_bwd(Hd, Wd, yd, md, old, ref, adv, w.n_resp, w.L, w.clip_eps, w.beta)
    lb, dHb, dWb = grpo.loss_fwd_bwd(Hp, Wd, yd, md, old, ref, adv, w.n_resp, w.L, w.clip_eps, w.beta)
    torch.cuda.synchronize()
    assert torch.equal(la, lb) and torch.equal(dHa, dHb) and torch.equal(dWa, dWb)


def test_host_hidden_states_inside_a_larger_pinned_allocation():
    """H as a view at an offset into a larger pinned buffer (the library maps the
    address of H itself, not the allocation's start)."""
    w = W_SMALL
    Hb, Wb, y, m, r, Hp = _inputs(w)
    big = torch.empty(w.T + 48, w.Hd, dtype=torch.bfloat16).pin_memory()
    big[48:] = Hp
    Hv = big[48:]
    assert Hv.is_pinned() and Hv.is_contiguous() and Hv.data_ptr() != big.data_ptr()
    Wd, yd, md = dev_tensor(Wb, torch.bfloat16), dev_tensor(y, torch.int32), dev_tensor(m, torch.uint8)
    assert torch.equal(grpo.token_logprobs(Hv, Wd, yd, md), grpo.token_logprobs(Hp, Wd, yd, md))


def test_pageable_host_hidden_states_are_copied_by_the_binding():
    """The binding copies pageable H to the device (the C ABI cannot read it)."""
    w = W_SMALL
    Hb, Wb, y, m, r, Hp = _inputs(w)
    Hpg = torch.from_numpy(np.ascontiguousarray(Hb)).view(torch.bfloat16)
    assert not Hpg.is_pinned()
    Wd, yd, md = dev_tensor(Wb, torch.bfloat16), dev_tensor(y, torch.int32), dev_tensor(m, torch.uint8)
    assert torch.equal(grpo.token_logprobs(Hpg, Wd, yd, md), grpo.token_logprobs(Hp, Wd, yd, md))


def test_c_abi_refuses_pageable_host_hidden_states():
    w = W_SMALL
    Hb, Wb, y, m, r, Hp = _inputs(w)
    Hnp = np.ascontiguousarray(Hb)                  # pageable numpy memory, 16-byte aligned by numpy
    assert Hnp.ctypes.data % 16 == 0
    Wd, yd, md = dev_tensor(Wb, torch.bfloat16), dev_tensor(y, torch.int32), dev_tensor(m, torch.uint8)
    out = torch.full((w.T,), 7.0, device=DEV)
    ws = grpo.workspace(w.T, w.Hd, w.V, grpo.GRPO_WS_LOGPROBS, DEV)
    lib = binding.load()
    st = lib.grpo_token_logprobs(ctypes.c_void_p(Hnp.ctypes.data), Wd.data_ptr(), yd.data_ptr(), md.data_ptr(),
                                 w.T, w.Hd, w.V, out.data_ptr(), ws.data_ptr(), ws.numel(),
                                 ctypes.c_void_p(torch.cuda.current_stream(DEV).cuda_stream))
    assert st == grpo.GRPO_ERR_INVALID_ARG
    torch.cuda.synchronize()
    assert bool((out == 7.0).all())                # nothing ran
    # the same call with the page-locked copy runs
    st = lib.grpo_token_logprobs(ctypes.c_void_p(Hp.data_ptr()), Wd.data_ptr(), yd.data_ptr(), md.data_ptr(),
                                 w.T, w.Hd, w.V, out.data_ptr(), ws.data_ptr(), ws.numel(),
                                 ctypes.c_void_p(torch.cuda.current_stream(DEV).cuda_stream))
    assert st == grpo.GRPO_OK
    assert torch.equal(out, grpo.token_logprobs(dev_tensor(Hb, torch.bfloat16), Wd, yd, md))
