#!/usr/bin/env python
"""Benchmark of the GRPO hot path on GB300.

One step = the group advantages (Eq. 2) followed by the fused log-prob, loss
and backward call (Eq. 1 and its gradient to H and W) over one synthetic batch
shaped like an 8B policy's rollout (workloads.py).  Prints one JSON line.

    python bench.py [--steps K] [--warmup W] [--workload fwdbwd_8b]
    python bench.py --impl reference ...      # the float64 CPU oracle, bounded sample
    torchrun --nproc-per-node N bench.py --gpus N ...

value: response (unmasked) tokens per second over all ranks, inputs resident
in HBM; e2e: the same through the public API with pinned host buffers, the
host<->device transfers inside the timed region.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import workloads as wl  # noqa: E402

METRIC = "response tokens/s for GRPO logprob+loss fwd+bwd; % of dense bf16 peak"
GOLDEN = {"fwdbwd_8b": "batch8b", "logprob3_8b": "batch8b", "long_8b": "long_8b", "ragged_8b": "ragged_8b"}
# the GEMM kernels, their launch parameters (raster, cache hints, chunk width)
# and the kept-logits dZ pass: what sets the DRAM traffic of the kernels the
# roofline reports
KERNEL_SOURCES = ["paper_2507_05687_gb300/csrc/gemm_tc.cuh", "paper_2507_05687_gb300/csrc/ptx.cuh",
                  "paper_2507_05687_gb300/csrc/gemm_launch.cuh", "paper_2507_05687_gb300/csrc/dz_rows.cuh"]
KIND_NAMES = ["advantages", "compact", "lse_gemm", "logp_merge", "loss", "dz_gemm", "dh_gemm", "dw_gemm",
              "dh_rows", "adamw", "sample_gemm", "transpose", "dz_logits", "top_p"]
# kernels per traced scope: compaction 4 (2 for batches of at most 4096 rows, whose mask
# count, scan and scatter run as one block), loss 2; others 1
KERNELS_PER_SCOPE = {1: 4, 4: 2}
SMALL_COMPACTION_ROWS = 4096


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=10)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default="fwdbwd_8b", choices=sorted(wl.ALL_WORKLOADS))
    p.add_argument("--adamw", choices=["none", "fused", "separate"], default="none",
                   help="fwd+bwd workloads: add the AdamW step of the LM head, fused into the dW GEMM "
                        "or as a separate pass over the stored dW")
    p.add_argument("--logits", choices=["keep", "recompute"], default="recompute",
                   help="fwd+bwd workloads: recompute the logits chunk by chunk in the backward with a second "
                        "logits GEMM, nothing of [tokens x vocabulary] size stored (GRPO_WS_LOSS, the default), "
                        "or keep the forward's fp32 logits for the backward (an exact GRPO_WS_LOSS_LOGITS workspace)")
    p.add_argument("--no-kept-compare", action="store_true",
                   help="skip the extra timing of the kept-logits backward reported beside the recomputing one")
    p.add_argument("--e2e-steps", type=int, default=20,
                   help="steps of the end-to-end measurement (per-step wall clock, median reported)")
    p.add_argument("--sample", action="store_true",
                   help="time the rollout draw (grpo_sample_tokens) over the workload's rows instead")
    p.add_argument("--top-p", type=float, default=1.0,
                   help="with --sample and a value below 1: the nucleus draw (grpo_sample_tokens_top_p), the "
                        "forward storing the logits and one selection pass per row")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--cpu-sample-tokens", type=int, default=1024,
                   help="tokens of the CPU-baseline sample (the reference arm uses a quarter per step)")
    return p.parse_args()


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return d["bf16_tflops"], d["bf16_tflops_sustained"], d["hbm_gbs"], "measured"
    except (OSError, KeyError, ValueError):
        return 1900.0, 1700.0, 6800.0, "fallback"


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


# ---------------------------------------------------------------- inputs

def make_inputs(w: wl.Workload):
    """Seeded host arrays of one batch, plus old/ref log-probs and where they came from."""
    Hb, Wb = wl.gen_hidden(w), wl.gen_weight(w)
    y, m, r = wl.gen_targets(w), wl.gen_mask(w), wl.gen_rewards(w)
    old = np.zeros(w.T, np.float32)
    ref = np.zeros(w.T, np.float32)
    src = lse_gold = None
    g = GOLDEN.get(w.name)
    path = os.path.join(ROOT, "tests", "golden", f"{g}.npz") if g else None
    if path and os.path.exists(path) and w.seed == wl.ALL_WORKLOADS[w.name].seed:
        d = np.load(path)
        idx = wl.valid_index(m)
        if int(d["n_valid"]) == idx.size:
            old[idx] = d["old_logp"]
            ref[idx] = d["ref_logp"]
            lse_gold = d["lse_policy"]
            src = "float64 oracle on the perturbed heads (tests/golden)"
    loss_gold = None
    lpath = os.path.join(ROOT, "tests", "golden", f"{g}_loss.json") if g else None
    if src is not None and lpath and os.path.exists(lpath):
        with open(lpath) as f:
            loss_gold = json.load(f)
        if loss_gold.get("workload") != w.name:
            loss_gold = None
    return dict(H=Hb, W=Wb, y=y, m=m, r=r, old=old, ref=ref, old_src=src, lse_gold=lse_gold, loss_gold=loss_gold)


def parity_loss(inp, loss_gpu: float, agg_mode: int = 0):
    """The library's loss of this batch against the float64 oracle's, stored by
    tests/golden/make_golden.py: the plain relative error and the error over
    max(|loss|, sum_t |w_t l_t|) (the advantages of a group sum to zero, so
    the loss can sit near 0 while its terms do not).  None without stored values."""
    gold = inp.get("loss_gold")
    if gold is None:
        return None
    want = gold[f"loss_agg{agg_mode}"]
    scale = max(abs(want), gold[f"sum_abs_terms_agg{agg_mode}"])
    d = abs(loss_gpu - want)
    return {"loss": loss_gpu, "loss_oracle": want, "loss_rel": d / abs(want) if want else None,
            "loss_rel_terms": d / scale, "loss_bar": 1e-3}


def parity_logp(inp, grpo, H, W, y, m):
    """The library's log-probs of this batch against the float64 oracle's, on every
    valid token: the oracle's log-sum-exp stored in tests/golden, minus nothing
    but the target logit recomputed here in float64 (one dot product per token).
    None when no stored values exist for the batch."""
    lse = inp.get("lse_gold")
    if lse is None:
        return None
    idx = wl.valid_index(inp["m"])
    got = grpo.token_logprobs(H, W, y, m).cpu().numpy()[idx].astype(np.float64)

    def widen(bits):
        return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)

    err = np.empty(idx.size)
    for a in range(0, idx.size, 8192):
        rows = idx[a:a + 8192]
        zy = np.einsum("ij,ij->i", widen(inp["H"][rows]), widen(inp["W"][inp["y"][rows]]))
        err[a:a + rows.size] = np.abs(got[a:a + rows.size] - (zy - lse[a:a + rows.size]))
    return {"logp_max_abs_err": float(err.max()), "logp_mean_abs_err": float(err.mean()), "tokens": int(idx.size),
            "bar": 2e-3, "reference": "float64 oracle (log-sum-exp stored in tests/golden, target logit in float64)"}


def fill_old_ref_on_gpu(w, inp, grpo, torch, dev):
    """old/ref log-probs of the perturbed heads from the library's own forward
    (what a GRPO pipeline does before the update); used when no stored oracle
    values exist for this batch."""
    Wold = wl.gen_weight(w, "old", inp["W"])
    Wref = wl.gen_weight(w, "ref", inp["W"])
    H = torch.from_numpy(inp["H"]).view(torch.bfloat16).to(dev)
    y = torch.from_numpy(inp["y"]).to(dev)
    m = torch.from_numpy(inp["m"]).to(dev)
    for key, Wx in (("old", Wold), ("ref", Wref)):
        lp = grpo.token_logprobs(H, torch.from_numpy(Wx).view(torch.bfloat16).to(dev), y, m)
        inp[key] = lp.cpu().numpy()
    inp["old_src"] = "library forward on the perturbed heads"


# ---------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi clock / throttle samples while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.out = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.out, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        self.proc.wait()
        self.out.flush()
        self.out.seek(0)
        rows = [l.strip().split(", ") for l in self.out if l.strip()]
        os.unlink(self.out.name)
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            try:
                sm.append(float(r[1]))
                mx = float(r[2])
                for n, v in zip(names, r[5:9]):
                    if v.strip().lower() == "active":
                        reasons.add(n)
            except (ValueError, IndexError):
                continue
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------- roofline

def kernel_hash() -> str:
    h = hashlib.sha256()
    for p in KERNEL_SOURCES:
        with open(os.path.join(ROOT, p), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


TRAFFIC_PATH = os.path.join(ROOT, "profiles", "traffic.txt")


def stored_traffic(variant: str, kind_name: str, Hd: int, V: int, n_valid: int, path: str = TRAFFIC_PATH):
    """DRAM bytes per launch of one kernel class, from a committed small-case ncu
    capture (profiles/traffic.txt lines '<hash> <variant> <capture workload>
    <capture rows> <kind> <bytes/launch> <cols/launch>'), scaled to n_valid
    rows: the capture runs the same kernel on the same hidden size and
    vocabulary over fewer rows, and each launch's operand panels, re-reads
    and outputs grow with its row tiles.  Only lines taken on the current
    kernel sources count.  Returns (bytes per launch at n_valid rows and the
    capture's columns, the capture's columns per launch, what was captured)
    or None."""
    if not os.path.exists(path):
        return None
    kh = kernel_hash()
    for line in open(path):
        f = line.split()
        if line.startswith("#") or len(f) < 7 or f[0] != kh or f[1] != variant or f[4] != kind_name:
            continue
        cw = wl.ALL_WORKLOADS.get(f[2])
        if cw is None or cw.Hd != Hd or cw.V != V:
            continue
        n_cap, b, cols = int(f[3]), float(f[5]), int(f[6])
        return b * n_valid / n_cap, cols, f"ncu on {f[2]} ({n_cap} unmasked rows), scaled by rows to {n_valid}"
    return None


def roofline(trace, n_valid_total_per_rank, Hd, steps, peak_tf, peak_kind, variant, hbm_gbs=None, V=None,
             traffic_path=TRAFFIC_PATH):
    by = {}
    for kind, cols, ms in trace:
        by.setdefault(kind, []).append((cols, ms))
    gemm_kinds = [2, 5, 6, 7, 10]
    dom = max(gemm_kinds, key=lambda k: sum(ms for _, ms in by.get(k, [])) if k in by else -1)
    recs = by[dom]
    flops = [2.0 * n_valid_total_per_rank * Hd * cols for cols, _ in recs]
    secs = [ms / 1e3 for _, ms in recs]
    achieved = (sum(flops) / len(flops)) / (sum(secs) / len(secs)) / 1e12
    total_ms = sum(ms for v in by.values() for _, ms in v)
    shares = {KIND_NAMES[k]: round(sum(ms for _, ms in v) / total_ms, 4) for k, v in sorted(by.items())}
    avg_cols = sum(c for c, _ in recs) / len(recs)
    tr = None if V is None else stored_traffic(variant, KIND_NAMES[dom], Hd, V, n_valid_total_per_rank,
                                               traffic_path)
    traffic = traffic_src = None
    if tr is not None:
        bytes_per_launch, cols_ref, traffic_src = tr
        traffic = bytes_per_launch * avg_cols / cols_ref
    common = {"kernel": KIND_NAMES[dom], "traffic": traffic, "traffic_from": traffic_src,
              "launches_per_step": len(recs) // max(1, steps),
              "avg_launch_ms": round(sum(secs) / len(secs) * 1e3, 4), "time_share": shares}
    if 13 in by and hbm_gbs:
        # nucleus selection + draw: the stored logits are read once from HBM per row
        # (the later passes over the row mostly hit L2): N_valid x V fp32 per launch
        tr13 = by[13]
        pb = 4.0 * n_valid_total_per_rank * (sum(c for c, _ in tr13) / len(tr13))
        ps = sum(ms for _, ms in tr13) / len(tr13) / 1e3
        common["top_p_hbm"] = {"achieved": round(pb / ps / 1e9, 1), "peak": hbm_gbs, "unit": "GB/s",
                               "frac": round(pb / ps / 1e9 / hbm_gbs, 4), "bytes_per_launch": pb,
                               "avg_launch_ms": round(ps * 1e3, 4)}
    if 12 in by and hbm_gbs:
        # dZ from the kept logits, HBM-bound: per launch it reads N_valid x cols
        # fp32 logits and writes N_valid x cols bf16 dZ (algorithmic bytes)
        zr = by[12]
        zb = sum(6.0 * n_valid_total_per_rank * c for c, _ in zr) / len(zr)
        zs = sum(ms for _, ms in zr) / len(zr) / 1e3
        ztr = None if V is None else stored_traffic(variant, "dz_logits", Hd, V, n_valid_total_per_rank,
                                                    traffic_path)
        common["dz_logits_hbm"] = {
            "achieved": round(zb / zs / 1e9, 1), "peak": hbm_gbs, "unit": "GB/s",
            "frac": round(zb / zs / 1e9 / hbm_gbs, 4), "bytes_per_launch": zb, "avg_launch_ms": round(zs * 1e3, 4),
            "traffic": None if ztr is None else ztr[0] * (sum(c for c, _ in zr) / len(zr)) / ztr[1]}
    # A forward launch over few rows (a decode step) reads all of W for little
    # work: below the ridge point (peak flop/s / peak B/s) its bound is HBM, and
    # its algorithmic bytes are W's columns plus the gathered rows.
    if hbm_gbs and dom in (2, 10):
        alg_bytes = 2.0 * Hd * avg_cols + 2.0 * Hd * n_valid_total_per_rank
        alg_flops = 2.0 * n_valid_total_per_rank * Hd * avg_cols
        if alg_flops / alg_bytes < peak_tf * 1e12 / (hbm_gbs * 1e9):
            gbs = alg_bytes / (sum(secs) / len(secs)) / 1e9
            return {"bound": "hbm", "achieved": round(gbs, 1), "peak": hbm_gbs,
                    "peak_kind": "HBM copy, measured", "unit": "GB/s", "frac": round(gbs / hbm_gbs, 4),
                    "bytes_per_launch": alg_bytes, **common}
    return {
        "bound": "tensor", "achieved": round(achieved, 1),
        "peak": peak_tf, "peak_kind": peak_kind, "unit": "TFLOP/s", "frac": round(achieved / peak_tf, 4),
        **common,
    }


# ---------------------------------------------------------------- CPU oracle

def cpu_oracle_sample(w, inp, n_tokens: int):
    """Times the float64 oracle's forward + backward on the first n_tokens
    unmasked tokens of the batch (whole responses from the start of the batch,
    full vocabulary and hidden size)."""
    import oracle
    L = w.L
    valid = np.flatnonzero(inp["m"])[:n_tokens]
    k = int(valid[-1] // L) + 1 if valid.size else 1
    m = np.zeros(k * L, np.uint8)
    m[valid] = 1
    adv = oracle.group_advantages(inp["r"], w.G, float(np.float32(w.adv_eps)))[:k]
    sl = slice(0, k * L)
    t0 = time.perf_counter()
    oracle.loss_fwd_bwd(inp["H"][sl], inp["W"], inp["y"][sl], m, inp["old"][sl], inp["ref"][sl], adv, k, L,
                        w.clip_eps, w.beta)
    dt = time.perf_counter() - t0
    return int(m.sum()), dt


def cpu_oracle_scoring_sample(w, inp, n_tokens: int):
    """Times the float64 oracle's log-probs of the first n_tokens unmasked tokens
    under the policy, old and reference heads (full vocabulary and hidden size)."""
    import oracle
    valid = np.flatnonzero(inp["m"])[:n_tokens]
    m = np.zeros(w.T, np.uint8)
    m[valid] = 1
    sl = slice(0, int(valid[-1]) + 1 if valid.size else 1)
    heads = [inp["W"], wl.gen_weight(w, "old", inp["W"]), wl.gen_weight(w, "ref", inp["W"])]
    t0 = time.perf_counter()
    for Wx in heads:
        oracle.token_logprobs(inp["H"][sl], Wx, inp["y"][sl], m[sl])
    return int(m.sum()), time.perf_counter() - t0


def run_reference(args):
    """The float64 oracle on the host cores, one bounded sample per step."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    w = wl.ALL_WORKLOADS[args.workload]
    inp = make_inputs(w)
    ntok = max(1, args.cpu_sample_tokens // 4)
    sample_fn = cpu_oracle_scoring_sample if w.name.startswith("logprob") else cpu_oracle_sample
    for _ in range(args.warmup):
        sample_fn(w, inp, ntok)
    toks, secs = 0, 0.0
    for _ in range(args.steps):
        n, dt = sample_fn(w, inp, ntok)
        toks += n
        secs += dt
    value = toks / secs
    sample = (f"first {toks // max(1, args.steps)} valid tokens of {w.name} per step: "
              f"oracle.loss_fwd_bwd in float64, full vocabulary and hidden size")
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 2), "unit": "tokens/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(secs / args.steps * 1e3, 1), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "sample": sample},
        "cpu_baseline": {"value": round(value, 2), "unit": "tokens/s", "cores": host_cores(), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": round(value, 2), "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------- GPU arm

def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
        return
    import torch

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)

    from paper_2507_05687_gb300 import build as build_mod
    build_mod.build()
    import paper_2507_05687_gb300 as grpo
    lib = grpo.load()

    base = wl.ALL_WORKLOADS[args.workload]
    w = base if rank == 0 else base.with_(seed=base.seed + 7919 * rank)
    sampling = args.sample  # the rollout draw over every unmasked row
    scoring = w.name.startswith("logprob") and not sampling  # log-probs of three heads, no loss / backward
    inp = make_inputs(w)
    if inp["old_src"] is None and not scoring and not sampling:
        fill_old_ref_on_gpu(w, inp, grpo, torch, dev)
    n_valid = int(inp["m"].sum())

    def to_dev(a, dt):
        return torch.from_numpy(np.ascontiguousarray(a)).view(dt).to(dev)

    H, W = to_dev(inp["H"], torch.bfloat16), to_dev(inp["W"], torch.bfloat16)
    y, m = to_dev(inp["y"], torch.int32), to_dev(inp["m"], torch.uint8)
    old, ref, r = to_dev(inp["old"], torch.float32), to_dev(inp["ref"], torch.float32), to_dev(inp["r"], torch.float32)
    from paper_2507_05687_gb300 import dp

    if sampling:
        top_p = args.top_p < 1.0
        ws = grpo.workspace(w.T, w.Hd, w.V, grpo.GRPO_WS_SAMPLE_TOP_P if top_p else grpo.GRPO_WS_SAMPLE, dev,
                            max_valid=n_valid)
        tok_out = (torch.empty(w.T, dtype=torch.int32, device=dev), torch.empty(w.T, dtype=torch.float32, device=dev))
        draw = [0]

        def step():
            draw[0] += 1  # a new offset per step: a fresh draw
            if top_p:
                grpo.sample_tokens_top_p(H, W, m, 1.0, args.top_p, seed=w.seed, offset=draw[0], ws=ws, out=tok_out)
            else:
                grpo.sample_tokens(H, W, m, 1.0, seed=w.seed, offset=draw[0], ws=ws, out=tok_out)
    elif scoring:
        heads = [W, to_dev(wl.gen_weight(w, "old", inp["W"]), torch.bfloat16),
                 to_dev(wl.gen_weight(w, "ref", inp["W"]), torch.bfloat16)]
        ws = grpo.workspace(w.T, w.Hd, w.V, grpo.GRPO_WS_LOGPROBS_HEADS, dev, max_valid=n_valid)
        logp3 = torch.empty(len(heads), w.T, dtype=torch.float32, device=dev)

        def step():
            # policy / old / reference log-probs of one rollout batch; ranks score independently
            grpo.token_logprobs_heads(H, heads, y, m, ws=ws, out=logp3)
    else:
        ws_kind = grpo.GRPO_WS_LOSS_LOGITS if args.logits == "keep" else grpo.GRPO_WS_LOSS
        ws = grpo.workspace(w.T, w.Hd, w.V, ws_kind, dev, max_valid=n_valid)
        if grpo.loss_plan(w.T, w.Hd, w.V, ws.numel())[0] != (args.logits == "keep"):
            raise SystemExit("the workspace does not give the requested logits handling")
        adv = torch.empty(w.n_resp, dtype=torch.float32, device=dev)
        out = (torch.empty(1, dtype=torch.float32, device=dev),
               torch.empty(w.T, w.Hd, dtype=torch.float32, device=dev),
               torch.empty(w.V, w.Hd, dtype=torch.float32, device=dev))

        if args.adamw != "none":
            master = W.float()
            exp_avg, exp_avg_sq = torch.zeros_like(master), torch.zeros_like(master)
            adam_step = [0]

        def step():
            grpo.group_advantages(r, w.G, w.adv_eps, out=adv)
            if args.adamw == "separate":
                adam_step[0] += 1
                grpo.loss_fwd_bwd(H, W, y, m, old, ref, adv, w.n_resp, w.L, w.clip_eps, w.beta, 0, ws=ws, out=out)
                grpo.adamw_step(master, exp_avg, exp_avg_sq, out[2], W, adam_step[0], lr=1e-6)
            elif args.adamw == "fused":
                # loss, dH and the actor's AdamW step on the LM head (lr 1e-6) in one call; dW is never stored
                adam_step[0] += 1
                norm = 0.0
                if dist is not None:
                    norm = dp.global_count(n_valid, dev)
                grpo.loss_fwd_bwd_adamw(H, W, y, m, old, ref, adv, w.n_resp, w.L, master, exp_avg, exp_avg_sq,
                                        adam_step[0], lr=1e-6, clip_eps=w.clip_eps, beta=w.beta, norm=norm, ws=ws,
                                        out=out[:2])
            elif dist is None:
                grpo.loss_fwd_bwd(H, W, y, m, old, ref, adv, w.n_resp, w.L, w.clip_eps, w.beta, 0, ws=ws, out=out)
            else:
                # global token-mean over every rank's batch; loss and dW summed over ranks
                dp.dp_loss_fwd_bwd(H, W, y, m, old, ref, adv, w.n_resp, w.L, w.clip_eps, w.beta, 0, n_valid,
                                   ws=ws, out=out)

    for _ in range(max(3, args.warmup)):
        step()
    st = grpo.check_device_status(ws)
    if st != grpo.GRPO_OK:
        raise SystemExit(f"device status after warm-up: {grpo.status_string(st)}")

    stream = torch.cuda.current_stream(dev)
    sampler = ClockSampler(local) if rank == 0 else None
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize(dev)
    if sampler:
        sampler.start()
    lib.grpo_trace_enable(1)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        step()
    ev1.record(stream)
    torch.cuda.synchronize(dev)
    lib.grpo_trace_enable(0)
    if dist is not None:
        dist.barrier()
    clocks = sampler.stop() if sampler else None
    ms = ev0.elapsed_time(ev1) / args.steps

    import ctypes
    nrec = lib.grpo_trace_read(None, None, None, 0)
    kinds = (ctypes.c_int32 * nrec)()
    cols = (ctypes.c_int64 * nrec)()
    kms = (ctypes.c_float * nrec)()
    lib.grpo_trace_read(kinds, cols, kms, nrec)
    trace = [(kinds[i], cols[i], kms[i]) for i in range(nrec)]
    per_scope = dict(KERNELS_PER_SCOPE)
    if w.T <= SMALL_COMPACTION_ROWS:
        per_scope[1] = 2
    launches = sum(per_scope.get(k, 1) for k, _, _ in trace)
    st = grpo.check_device_status(ws)
    if st != grpo.GRPO_OK:
        raise SystemExit(f"device status after timing: {grpo.status_string(st)}")

    loss_timed = None if sampling or scoring or args.adamw != "none" else float(out[0].item())
    tot_valid = n_valid
    if dist is not None:
        t = torch.tensor([ms], device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = t.item()
        n = torch.tensor([n_valid], device=dev, dtype=torch.float64)
        dist.all_reduce(n)
        tot_valid = int(n.item())
    value = tot_valid / (ms / 1e3)

    burst, sustained, hbm, peak_src = peaks()
    rf = roofline(trace, n_valid, w.Hd, args.steps, sustained, f"bf16 sustained, {peak_src}",
                  path_variant(args, sampling, scoring), hbm, V=w.V)
    if sampling:
        step_exec = step_model = 2.0 * n_valid * w.Hd * w.V
    elif scoring:
        step_exec = step_model = 2.0 * 3 * n_valid * w.Hd * w.V  # three forward passes, nothing recomputed
    else:
        # executed GEMM flops: forward, dH, dW, plus the recomputed logits GEMM
        # when the logits are not kept; the textbook count is forward + backward
        step_exec = (6.0 if args.logits == "keep" else 8.0) * n_valid * w.Hd * w.V
        step_model = 6.0 * n_valid * w.Hd * w.V

    e2e = e2e_offload = e2e_staged = None
    if not args.no_e2e and not sampling:
        if scoring:
            e2e = measure_e2e_scoring(grpo, torch, dev, w, inp, heads, steps=args.e2e_steps, dist=dist)
        else:
            # the step's own workspace: a second one of the same size may not fit beside it
            e2e = measure_e2e(grpo, torch, dev, w, inp, steps=args.e2e_steps, dist=dist, ws=ws)
            if dist is None:
                e2e_staged = measure_e2e_staged(grpo, torch, dev, w, inp, steps=args.e2e_steps, ws=ws)
            if world == 1:
                e2e_offload = measure_e2e_offload(grpo, torch, dev, w, inp, steps=args.e2e_steps, ws=ws)

    kept = None
    if not (args.no_kept_compare or sampling or scoring) and args.logits == "recompute" and args.adamw == "none" \
            and world == 1:
        kept = measure_kept_logits(grpo, torch, dev, w, (H, W, y, m, old, ref, r), n_valid,
                                   steps=min(args.steps, 10), out=out)

    parity = None
    if rank == 0 and not sampling:
        parity = parity_logp(inp, grpo, H, W, y, m) or {}
        if loss_timed is not None and world == 1:
            parity.update(parity_loss(inp, loss_timed) or {})
        parity = parity or None

    cpu = None
    if not args.no_cpu_baseline and rank == 0 and world == 1 and not sampling:
        ntok, dt = (cpu_oracle_scoring_sample if scoring else cpu_oracle_sample)(w, inp, args.cpu_sample_tokens)
        cpu = {"value": round(ntok / dt, 2), "unit": "tokens/s", "cores": host_cores(), "kind": "oracle",
               "sample": f"first {ntok} valid tokens of {w.name}: "
                         f"{'oracle.token_logprobs under 3 heads' if scoring else 'oracle.loss_fwd_bwd'} in "
                         f"float64 over the full vocabulary and hidden size, {dt:.1f} s"}

    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 1), "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": max(3, args.warmup), "ms_per_step": round(ms, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic",
            "config": {"workload": w.name, "prompts": w.n_prompts, "G": w.G, "L": w.L, "Hd": w.Hd, "V": w.V,
                       "tokens": w.T, "n_valid": n_valid, "global_valid_tokens": tot_valid,
                       "parallelism": f"dp{world}",
                       "l2": "inputs larger than L2 (W %.2f GB, H %.2f GB per rank)" % (w.V * w.Hd * 2 / 1e9,
                                                                                         w.T * w.Hd * 2 / 1e9),
                       "old_ref_logp": inp["old_src"], "adamw": args.adamw,
                       "logits": None if sampling or scoring else
                       ("kept from the forward" if args.logits == "keep" else "recomputed in the backward"),
                       "step": "sample" if sampling else ("score3" if scoring else "fwdbwd"),
                       "top_p": args.top_p if sampling else None},
            "step_gemm_tflops_executed": round(step_exec / (ms / 1e3) / 1e12, 1),
            "step_frac_executed": round(step_exec / (ms / 1e3) / 1e12 / burst, 4),
            "step_frac_6x": round(step_model / (ms / 1e3) / 1e12 / burst, 4),
            "roofline": rf, "clocks": clocks, "gpu_launches": launches, "e2e": e2e, "cpu_baseline": cpu,
            "parity": parity,
        }
        if e2e_offload is not None:
            line["e2e_offload"] = e2e_offload
        if e2e_staged is not None:
            line["e2e_staged"] = e2e_staged
        if kept is not None:
            line["kept_logits_ms_per_step"] = kept.get("ms_per_step")
            line["kept_logits"] = kept
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


def path_variant(args, sampling: bool, scoring: bool) -> str:
    """Which code path a run times (the key of its traffic lines)."""
    if sampling:
        return "sample" + ("+top_p" if args.top_p < 1.0 else "")
    if scoring:
        return "score3"
    return "fwdbwd" + ("+kept" if args.logits == "keep" else "") + \
        ("" if args.adamw == "none" else "+adamw_" + args.adamw)


def measure_kept_logits(grpo, torch, dev, w, tensors, n_valid: int, steps: int, out):
    """The same step with the opt-in backward that keeps the forward's fp32
    logits (an exact GRPO_WS_LOSS_LOGITS workspace for the unmasked rows):
    timed like the main step, reported beside it.  None (with the reason) when
    that workspace does not fit in the free device memory."""
    H, W, y, m, old, ref, r = tensors
    need = grpo.workspace_bytes_rows(w.T, n_valid, w.Hd, w.V, grpo.GRPO_WS_LOSS_LOGITS)
    torch.cuda.empty_cache()
    free = torch.cuda.mem_get_info(dev)[0]
    if need > free - (2 << 30):
        return {"ms_per_step": None, "skipped": f"workspace of {need / 1e9:.1f} GB does not fit ({free / 1e9:.1f} GB free)"}
    ws = grpo.workspace(w.T, w.Hd, w.V, grpo.GRPO_WS_LOSS_LOGITS, dev, max_valid=n_valid)
    if grpo.loss_plan(w.T, w.Hd, w.V, ws.numel())[0] != 1:
        raise SystemExit("the kept-logits workspace does not keep the logits")
    adv = torch.empty(w.n_resp, dtype=torch.float32, device=dev)

    def step():
        grpo.group_advantages(r, w.G, w.adv_eps, out=adv)
        grpo.loss_fwd_bwd(H, W, y, m, old, ref, adv, w.n_resp, w.L, w.clip_eps, w.beta, 0, ws=ws, out=out)

    for _ in range(3):
        step()
    if grpo.check_device_status(ws) != grpo.GRPO_OK:
        raise SystemExit("device status after the kept-logits warm-up is not OK")
    stream = torch.cuda.current_stream(dev)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize(dev)
    ev0.record(stream)
    for _ in range(steps):
        step()
    ev1.record(stream)
    torch.cuda.synchronize(dev)
    ms = ev0.elapsed_time(ev1) / steps
    st = grpo.check_device_status(ws)
    del ws
    torch.cuda.empty_cache()
    if st != grpo.GRPO_OK:
        raise SystemExit("device status after the kept-logits steps is not OK")
    return {"ms_per_step": round(ms, 3), "value": round(n_valid / (ms / 1e3), 1), "unit": "tokens/s",
            "steps": steps, "workspace_bytes": int(need),
            "what": "opt-in variant: the forward stores the fp32 logits [rows x V] in the workspace and the "
                    "backward forms dZ from them by an HBM pass instead of the recomputing GEMM"}


def timed_steps(one, steps: int):
    """(median, mean) wall-clock seconds of `steps` calls of one(), each of which
    returns only once its results are on the host."""
    ts = []
    for _ in range(max(1, steps)):
        t0 = time.perf_counter()
        one()
        ts.append(time.perf_counter() - t0)
    return statistics.median(ts), sum(ts) / len(ts)


def across_ranks(torch, dev, dist, dt: float, n_tok: int):
    """(slowest rank's seconds per step, tokens summed over ranks)."""
    if dist is None:
        return dt, n_tok
    t = torch.tensor([dt, float(n_tok)], dtype=torch.float64, device=dev)
    dist.all_reduce(t[:1], op=dist.ReduceOp.MAX)
    dist.all_reduce(t[1:], op=dist.ReduceOp.SUM)
    return float(t[0].item()), int(t[1].item())


def measure_e2e_scoring(grpo, torch, dev, w, inp, heads, steps: int, dist=None):
    """Public API, rollout scoring: H2D of the batch (H, targets, mask) from pinned host
    memory, the three LM heads resident on the device (model weights), D2H of the
    three log-prob rows.  Across ranks each scores its own batch (no exchange);
    the time is the slowest rank's and the tokens are summed."""
    n_valid = int(inp["m"].sum())

    def pin(a, dt):
        return torch.from_numpy(np.ascontiguousarray(a)).view(dt).pin_memory()

    hH, hy, hm = pin(inp["H"], torch.bfloat16), pin(inp["y"], torch.int32), pin(inp["m"], torch.uint8)
    # H stays in page-locked host memory: the row gather reads the unmasked rows over the host link
    h2d = n_valid * w.Hd * 2 + sum(t.numel() * t.element_size() for t in [hy, hm])
    d2h = len(heads) * w.T * 4
    hout = torch.empty(len(heads), w.T, dtype=torch.float32).pin_memory()
    ws = grpo.workspace(w.T, w.Hd, w.V, grpo.GRPO_WS_LOGPROBS_HEADS, dev, max_valid=n_valid)

    def one():
        lp = grpo.token_logprobs_heads(hH, heads, hy, hm, ws=ws)
        hout.copy_(lp, non_blocking=True)
        torch.cuda.current_stream(dev).synchronize()

    one()
    if dist is not None:
        dist.barrier()
    med, mean = timed_steps(one, steps)
    dt, n_tok = across_ranks(torch, dev, dist, med, n_valid)
    return {"value": round(n_tok / dt, 1), "unit": "tokens/s", "ms_per_step": round(dt * 1e3, 2),
            "ms_mean": round(mean * 1e3, 2), "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "steps": steps, "statistic": "median of per-step wall-clock times",
            "what": "H read from pinned host memory by the row gather each step (the unmasked rows cross the "
                    "host link), targets and mask copied; the policy / old / reference heads resident on the "
                    "device; the log-probs read back"}


def measure_e2e(grpo, torch, dev, w, inp, steps: int, dist=None, ws=None):
    """Public API, one training step: H2D of the batch (H, targets, mask, old / ref
    log-probs, rewards) from pinned host memory, the LM head W resident on the
    device (the parameter being trained), D2H of the loss; dH and dW stay on the
    device, where the trunk's backward and the optimiser consume them.  Across
    ranks every rank runs the data-parallel call on its own batch; the time is
    the slowest rank's and the tokens are summed, like the device-timed value."""
    from paper_2507_05687_gb300 import dp
    n_valid = int(inp["m"].sum())

    def pin(a, dt):
        return torch.from_numpy(np.ascontiguousarray(a)).view(dt).pin_memory()

    Wd = torch.from_numpy(np.ascontiguousarray(inp["W"])).view(torch.bfloat16).to(dev)
    hH, hy, hm = pin(inp["H"], torch.bfloat16), pin(inp["y"], torch.int32), pin(inp["m"], torch.uint8)
    hold, href, hr = pin(inp["old"], torch.float32), pin(inp["ref"], torch.float32), pin(inp["r"], torch.float32)
    # H stays in page-locked host memory: the row gather reads the unmasked rows over the host link
    h2d = n_valid * w.Hd * 2 + sum(t.numel() * t.element_size() for t in (hy, hm, hold, href, hr))
    d2h = 4
    out = (torch.empty(1, dtype=torch.float32, device=dev), torch.empty(w.T, w.Hd, dtype=torch.float32, device=dev),
           torch.empty(w.V, w.Hd, dtype=torch.float32, device=dev))
    if ws is None:
        ws = grpo.loss_workspace(w.T, w.Hd, w.V, dev, max_valid=n_valid)

    def one():
        adv = grpo.group_advantages(hr.to(dev, non_blocking=True), w.G, w.adv_eps)
        if dist is None:
            loss, _, _ = grpo.loss_fwd_bwd(hH, Wd, hy, hm, hold, href, adv, w.n_resp, w.L, w.clip_eps, w.beta,
                                           ws=ws, out=out)
        else:
            loss, _, _ = dp.dp_loss_fwd_bwd(hH, Wd, hy, hm, hold, href, adv, w.n_resp, w.L, w.clip_eps, w.beta, 0,
                                            n_valid, ws=ws, out=out)
        return loss.item()

    one()
    torch.cuda.synchronize(dev)
    if dist is not None:
        dist.barrier()
    med, mean = timed_steps(one, steps)
    dt, n_tok = across_ranks(torch, dev, dist, med, n_valid)
    return {"value": round(n_tok / dt, 1), "unit": "tokens/s", "ms_per_step": round(dt * 1e3, 2),
            "ms_mean": round(mean * 1e3, 2), "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "steps": steps, "statistic": "median of per-step wall-clock times",
            "what": "H read from pinned host memory by the row gather each step (the unmasked rows cross the "
                    "host link); targets, mask, old/ref log-probs, rewards copied; W resident on the device; the "
                    "loss read back; dH, dW left on the device"}


def measure_e2e_staged(grpo, torch, dev, w, inp, steps: int, ws=None):
    """The training step of measure_e2e fed through staging.BatchStager: each
    step's whole batch (every row of H, targets, mask, old / ref log-probs,
    rewards) is copied from pinned host memory into a device slot on a copy
    stream while the previous step computes; the step waits for its batch's
    copies, runs on the device tensors and reads the loss back."""
    from paper_2507_05687_gb300.staging import BatchStager
    n_valid = int(inp["m"].sum())

    def pin(a, dt):
        return torch.from_numpy(np.ascontiguousarray(a)).view(dt).pin_memory()

    Wd = torch.from_numpy(np.ascontiguousarray(inp["W"])).view(torch.bfloat16).to(dev)
    batch = (pin(inp["H"], torch.bfloat16), pin(inp["y"], torch.int32), pin(inp["m"], torch.uint8),
             pin(inp["old"], torch.float32), pin(inp["ref"], torch.float32), pin(inp["r"], torch.float32))
    h2d = sum(t.numel() * t.element_size() for t in batch)
    out = (torch.empty(1, dtype=torch.float32, device=dev), torch.empty(w.T, w.Hd, dtype=torch.float32, device=dev),
           torch.empty(w.V, w.Hd, dtype=torch.float32, device=dev))
    if ws is None:
        ws = grpo.loss_workspace(w.T, w.Hd, w.V, dev, max_valid=n_valid)
    stager = BatchStager(dev)
    stager.submit(batch)

    def one():
        H, y, m, old, ref, r = stager.get()
        stager.submit(batch)  # the next step's batch (the same synthetic arrays), copied while this one runs
        adv = grpo.group_advantages(r, w.G, w.adv_eps)
        loss, _, _ = grpo.loss_fwd_bwd(H, Wd, y, m, old, ref, adv, w.n_resp, w.L, w.clip_eps, w.beta, ws=ws, out=out)
        stager.release()
        return loss.item()

    one()
    torch.cuda.synchronize(dev)
    med, mean = timed_steps(one, steps)
    return {"value": round(n_valid / med, 1), "unit": "tokens/s", "ms_per_step": round(med * 1e3, 2),
            "ms_mean": round(mean * 1e3, 2), "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": 4,
            "steps": steps, "statistic": "median of per-step wall-clock times",
            "what": "the whole batch copied from pinned host memory each step on a copy stream while the previous "
                    "step computes (staging.BatchStager, two device slots); the step waits for its copies; W "
                    "resident; the loss read back"}


def measure_e2e_offload(grpo, torch, dev, w, inp, steps: int, ws=None):
    """Public API with everything on the host (a host-offloaded head): H2D of the
    batch and of W, the step, D2H of loss, dH, dW (dW streamed chunk by chunk)."""
    n_valid = int(inp["m"].sum())

    def pin(a, dt):
        t = torch.from_numpy(np.ascontiguousarray(a)).view(dt)
        return t.pin_memory()

    hH, hW = pin(inp["H"], torch.bfloat16), pin(inp["W"], torch.bfloat16)
    hy, hm = pin(inp["y"], torch.int32), pin(inp["m"], torch.uint8)
    hold, href, hr = pin(inp["old"], torch.float32), pin(inp["ref"], torch.float32), pin(inp["r"], torch.float32)
    # H stays in page-locked host memory (the row gather reads the unmasked rows); W is copied
    h2d = n_valid * w.Hd * 2 + sum(t.numel() * t.element_size() for t in (hW, hy, hm, hold, href, hr))
    d2h = 4 + w.T * w.Hd * 4 + w.V * w.Hd * 4

    # the caller's own buffers, allocated once: pinned host outputs and a device workspace
    hout = (torch.empty(1, dtype=torch.float32).pin_memory(), torch.empty(w.T, w.Hd, dtype=torch.float32).pin_memory(),
            torch.empty(w.V, w.Hd, dtype=torch.float32).pin_memory())
    if ws is None:
        ws = grpo.loss_workspace(w.T, w.Hd, w.V, dev, max_valid=n_valid)

    def one():
        adv = grpo.group_advantages(hr.to(dev, non_blocking=True), w.G, w.adv_eps)
        return grpo.loss_fwd_bwd(hH, hW, hy, hm, hold, href, adv, w.n_resp, w.L, w.clip_eps, w.beta, ws=ws, out=hout)

    one()
    torch.cuda.synchronize(dev)
    med, mean = timed_steps(one, steps)   # one() returns pinned host tensors once they have landed
    return {"value": round(n_valid / med, 1), "unit": "tokens/s", "ms_per_step": round(med * 1e3, 2),
            "ms_mean": round(mean * 1e3, 2), "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "steps": steps, "statistic": "median of per-step wall-clock times",
            "what": "H read from pinned host memory by the row gather (the unmasked rows cross the host link); "
                    "the rest of the batch and W copied each step; loss, dH, dW copied back"}


if __name__ == "__main__":
    main()
