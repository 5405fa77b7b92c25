"""Seeded synthetic GRPO workloads: shapes, seeds and value distributions.

This module is shared by the tests, ``bench.py`` and ``__graft_entry__.smoke``.
It holds random draws, integer bookkeeping and bf16 rounding of the draws only;
none of the GRPO arithmetic (Eq. 1, Eq. 2) lives here.  Both the float64 oracle
and the CUDA path are fed the arrays it returns, so they see bit-identical
inputs.

Every array has its own PCG64 stream keyed by (seed, stream id, chunk index),
with a fixed chunking, so the values do not depend on the number of threads
used to draw them and are the same on x86_64 and aarch64 hosts.

Value recipe (the 8B-shaped workloads follow the paper's backbone and RL
setup, Section 3.3 and Section 4.1: 64 prompts per step, long responses):

* hidden states H  [T, Hd]  ~ N(0, 1), rounded to bf16 (round-to-nearest-even)
* policy LM head W [V, Hd]  ~ N(0, 0.02), bf16
* old policy       W + N(0, 0.002), rounded to bf16
* reference policy W + N(0, 0.004), rounded to bf16
* targets y_t ~ U{0 .. V-1}
* response lengths: all L, U{lo..hi} or log-uniform on [lo, hi]; the mask is a
  prefix of each response's L padded rows
* rewards: Bernoulli(0.3) in {0, 1}, or 0.5*Bern(0.3) + 0.5*Bern(0.2); some
  groups can be forced to equal rewards (the zero-std advantage case)
"""
from __future__ import annotations

import math
import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, replace

import numpy as np

SEED_BASE = 250705687

# Stream identifiers: one independent PCG64 stream family per array.
_S_LEN, _S_MASK, _S_TGT, _S_REW, _S_H, _S_W, _S_OLD, _S_REF, _S_ZSTD = range(1, 10)
_ROWS_PER_CHUNK = 1024


@dataclass(frozen=True)
class Workload:
    """One synthetic GRPO batch.

    Token layout is padded: response i owns rows [i*L, (i+1)*L) of H, targets
    and mask; responses of one prompt group are contiguous runs of G.
    """

    name: str
    n_prompts: int
    G: int
    L: int
    Hd: int
    V: int
    lengths: str = "full"      # "full" | "uniform" | "loguniform"
    len_lo: int = 0
    len_hi: int = 0
    rewards: str = "bern"      # "bern" (Bern(0.3)) | "mix" (0.5 Bern(0.3) + 0.5 Bern(0.2))
    zero_std_every: int = 0    # every k-th group gets all-equal rewards (0: none)
    seed: int = SEED_BASE
    clip_eps: float = 0.2
    beta: float = 0.04
    adv_eps: float = 1e-6
    h_std: float = 1.0
    w_std: float = 0.02
    old_std: float = 0.002
    ref_std: float = 0.004

    @property
    def n_resp(self) -> int:
        return self.n_prompts * self.G

    @property
    def T(self) -> int:
        return self.n_resp * self.L

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


# The five workloads: a tiny oracle-scale batch and four shaped like an 8B
# policy (hidden 4096, vocabulary 155136).
WORKLOADS = {
    # seed: the first of SEED_BASE + 1, + 11, ... whose Bern(0.3) group is not all-equal
    "tiny_fwdbwd": Workload("tiny_fwdbwd", 1, 4, 64, 256, 4096, seed=SEED_BASE + 11),
    "logprob3_8b": Workload("logprob3_8b", 8, 8, 512, 4096, 155136, "uniform", 128, 512,
                            seed=SEED_BASE + 2),
    # same 32768-token batch as logprob3_8b (same seed), mixed rewards
    "fwdbwd_8b": Workload("fwdbwd_8b", 8, 8, 512, 4096, 155136, "uniform", 128, 512,
                          rewards="mix", seed=SEED_BASE + 2),
    "long_8b": Workload("long_8b", 4, 16, 4096, 4096, 155136, "uniform", 1024, 4096,
                        rewards="mix", seed=SEED_BASE + 4),
    "ragged_8b": Workload("ragged_8b", 16, 8, 8192, 4096, 155136, "loguniform", 16, 8192,
                          rewards="mix", zero_std_every=4, seed=SEED_BASE + 5),
}

# Smaller cases of the same kernels, for profiler captures that must stay a
# few GB on the device (inputs still larger than the 129 MB L2).
PROFILE_WORKLOADS = {
    "fwdbwd_small": Workload("fwdbwd_small", 2, 8, 512, 4096, 32768, "uniform", 128, 512,
                             rewards="mix", seed=SEED_BASE + 6),
    # the bench's hidden size, vocabulary, vocabulary chunks and lengths over a
    # quarter of its prompts (about 5k unmasked rows, about 5 GB on the device):
    # DRAM-counter captures of single GEMM launches, scaled to the bench by rows
    "fwdbwd_mid": Workload("fwdbwd_mid", 2, 8, 512, 4096, 155136, "uniform", 128, 512,
                           rewards="mix", seed=SEED_BASE + 8),
}
# One decode step of rollout generation: every active sequence samples its next
# token, so the LM-head GEMM sees a few hundred to a few thousand rows (here
# 64 prompts x G=8 sequences = 512 rows, and 256 / 2048 rows), one per sequence.
DECODE_WORKLOADS = {
    "decode256_8b": Workload("decode256_8b", 32, 8, 1, 4096, 155136, seed=SEED_BASE + 7),
    "decode512_8b": Workload("decode512_8b", 64, 8, 1, 4096, 155136, seed=SEED_BASE + 7),
    "decode2048_8b": Workload("decode2048_8b", 256, 8, 1, 4096, 155136, seed=SEED_BASE + 7),
}
ALL_WORKLOADS = {**WORKLOADS, **PROFILE_WORKLOADS, **DECODE_WORKLOADS}


def _rng(seed: int, stream: int, chunk: int = 0) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, stream, chunk])))


def _threads() -> int:
    try:
        n = len(os.sched_getaffinity(0))
    except AttributeError:  # pragma: no cover
        n = os.cpu_count() or 1
    return max(1, min(32, n))


# ---------------------------------------------------------------------------
# bf16 rounding of the draws (storage format of H and W)
# ---------------------------------------------------------------------------

def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (nearest, ties to even); returns the uint16 bit patterns."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    r = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32."""
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


# ---------------------------------------------------------------------------
# integer parts: lengths, mask, targets, rewards
# ---------------------------------------------------------------------------

def gen_lengths(w: Workload) -> np.ndarray:
    """Unpadded length |o_i| of every response, int64 [n_resp]."""
    rng = _rng(w.seed, _S_LEN)
    if w.lengths == "full":
        return np.full(w.n_resp, w.L, dtype=np.int64)
    if w.lengths == "uniform":
        return rng.integers(w.len_lo, w.len_hi, size=w.n_resp, endpoint=True).astype(np.int64)
    if w.lengths == "loguniform":
        u = rng.random(w.n_resp)
        x = np.exp(math.log(w.len_lo) + u * (math.log(w.len_hi) - math.log(w.len_lo)))
        return np.clip(np.floor(x), w.len_lo, w.len_hi).astype(np.int64)
    raise ValueError(w.lengths)


def gen_mask(w: Workload, lengths: np.ndarray | None = None) -> np.ndarray:
    """uint8 [T]; row i*L + j is 1 iff j < |o_i| (a prefix of each response)."""
    if lengths is None:
        lengths = gen_lengths(w)
    j = np.arange(w.L, dtype=np.int64)[None, :]
    return (j < lengths[:, None]).astype(np.uint8).reshape(-1)


def gen_targets(w: Workload) -> np.ndarray:
    """int32 [T], the sampled token at every row, uniform on [0, V)."""
    out = np.empty(w.T, dtype=np.int32)
    n = (w.T + _ROWS_PER_CHUNK * 64 - 1) // (_ROWS_PER_CHUNK * 64)
    step = _ROWS_PER_CHUNK * 64
    for c in range(n):
        lo, hi = c * step, min(w.T, (c + 1) * step)
        out[lo:hi] = _rng(w.seed, _S_TGT, c).integers(0, w.V, size=hi - lo, dtype=np.int32)
    return out


def gen_rewards(w: Workload) -> np.ndarray:
    """float32 [n_resp] rewards (synthetic stand-in for the Eq. 3 reward)."""
    rng = _rng(w.seed, _S_REW)
    if w.rewards == "bern":
        r = (rng.random(w.n_resp) < 0.3).astype(np.float32)
    elif w.rewards == "mix":
        a = (rng.random(w.n_resp) < 0.3).astype(np.float32)
        b = (rng.random(w.n_resp) < 0.2).astype(np.float32)
        r = (np.float32(0.5) * a + np.float32(0.5) * b).astype(np.float32)
    else:
        raise ValueError(w.rewards)
    if w.zero_std_every:
        r = r.reshape(w.n_prompts, w.G).copy()
        for g in range(0, w.n_prompts, w.zero_std_every):
            r[g, :] = r[g, 0]
        r = r.reshape(-1)
    return r


# ---------------------------------------------------------------------------
# floating parts: hidden states and LM-head weights (bf16 bit patterns)
# ---------------------------------------------------------------------------

def _normal_rows_bf16(seed: int, stream: int, rows: int, cols: int, std: float,
                      base: np.ndarray | None = None) -> np.ndarray:
    """bf16 bits of std*N(0,1) (+ widened base), drawn in fixed 1024-row chunks."""
    out = np.empty((rows, cols), dtype=np.uint16)
    nchunk = (rows + _ROWS_PER_CHUNK - 1) // _ROWS_PER_CHUNK

    def work(c: int) -> None:
        lo, hi = c * _ROWS_PER_CHUNK, min(rows, (c + 1) * _ROWS_PER_CHUNK)
        x = _rng(seed, stream, c).standard_normal((hi - lo, cols), dtype=np.float32)
        x *= np.float32(std)
        if base is not None:
            x += bf16_bits_to_f32(base[lo:hi])
        out[lo:hi] = f32_to_bf16_bits(x)

    with ThreadPoolExecutor(_threads()) as ex:
        list(ex.map(work, range(nchunk)))
    return out


def gen_hidden(w: Workload) -> np.ndarray:
    """bf16 bits [T, Hd] of the policy's final hidden states (padded rows included)."""
    return _normal_rows_bf16(w.seed, _S_H, w.T, w.Hd, w.h_std)


def gen_weight(w: Workload, which: str = "policy", policy: np.ndarray | None = None) -> np.ndarray:
    """bf16 bits [V, Hd] of an LM-head weight: 'policy', 'old' or 'ref'."""
    if which == "policy":
        return _normal_rows_bf16(w.seed, _S_W, w.V, w.Hd, w.w_std)
    if policy is None:
        policy = gen_weight(w, "policy")
    if which == "old":
        return _normal_rows_bf16(w.seed, _S_OLD, w.V, w.Hd, w.old_std, base=policy)
    if which == "ref":
        return _normal_rows_bf16(w.seed, _S_REF, w.V, w.Hd, w.ref_std, base=policy)
    raise ValueError(which)


def valid_index(mask: np.ndarray) -> np.ndarray:
    """Positions of the unmasked rows in increasing order (int64)."""
    return np.flatnonzero(np.asarray(mask) != 0).astype(np.int64)


def sample_rows(n: int, k: int, seed: int, must: np.ndarray | None = None) -> np.ndarray:
    """A sorted seeded sample of k distinct indices in [0, n), plus the 'must' ones."""
    rng = _rng(seed, 99)
    k = min(k, n)
    s = rng.choice(n, size=k, replace=False) if k else np.zeros(0, dtype=np.int64)
    if must is not None and len(must):
        s = np.concatenate([s, np.asarray(must, dtype=np.int64)])
    return np.unique(s.astype(np.int64))
