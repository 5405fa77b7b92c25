"""Data-parallel host logic on CPU ranks (gloo, world size 2).

Each rank owns whole prompt groups and computes its shard with the float64
oracle; paper_2507_05687_gb300.dp supplies the global normaliser and the sum
of loss and dW.  The result must equal the oracle on the whole batch.  A rank
that fails before the collective must make the other rank raise (a short
process-group timeout), not hang.
"""
import datetime
import multiprocessing as mp
import os
import socket
import traceback

import numpy as np
import pytest

from paper_2507_05687_gb300 import dp

torch = pytest.importorskip("torch")


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_shard_groups_cover_every_group_once():
    for n in (0, 1, 5, 8, 13, 64):
        for world in (1, 2, 3, 8):
            spans = [dp.shard_groups(n, world, r) for r in range(world)]
            assert spans[0][0] == 0 and spans[-1][1] == n
            for (a0, a1), (b0, b1) in zip(spans, spans[1:]):
                assert a1 == b0
            sizes = [b - a for a, b in spans]
            assert max(sizes) - min(sizes) <= 1
    with pytest.raises(ValueError):
        dp.shard_groups(4, 2, 2)
    rs, ts = dp.shard_rows(5, 4, 10, 2, 1)
    assert (rs.start, rs.stop, ts.start, ts.stop) == (12, 20, 120, 200)


def test_chunk_rows_cover_every_vocabulary_row_once():
    for V in (1, 255, 256, 4097, 155136):
        for cols in (256, 768, 16384):
            rows = dp.chunk_rows(V, cols)
            assert rows[0].start == 0 and rows[-1].stop == V
            assert all(a.stop == b.start for a, b in zip(rows, rows[1:]))
            assert all(0 < r.stop - r.start <= cols for r in rows)
            assert len(rows) == -(-V // cols)
    assert dp.chunk_rows(10, 0) == []


def _batch():
    import oracle
    import workloads as wl
    w = wl.Workload("dp", 5, 2, 6, 8, 11, "uniform", 1, 6, rewards="mix", seed=wl.SEED_BASE + 31337, w_std=0.7)
    H, W = oracle.widen_bf16(wl.gen_hidden(w)), oracle.widen_bf16(wl.gen_weight(w))
    y, m, r = wl.gen_targets(w), wl.gen_mask(w), wl.gen_rewards(w)
    old = oracle.token_logprobs(H, oracle.widen_bf16(wl.gen_weight(w, "old", wl.gen_weight(w))), y, m)[0]
    ref = oracle.token_logprobs(H, oracle.widen_bf16(wl.gen_weight(w, "ref", wl.gen_weight(w))), y, m)[0]
    adv = oracle.group_advantages(r, w.G)
    return w, H, W, y, m, old, ref, adv


def _oracle_compute(H, W, y, m, old, ref, adv, n_resp, L, clip, beta, agg, norm):
    import oracle
    out = oracle.loss_fwd_bwd(H, W, y, m, old, ref, adv, n_resp, L, clip, beta, agg, norm=norm)
    return (torch.tensor([out["loss"]], dtype=torch.float64), torch.from_numpy(out["dH"]),
            torch.from_numpy(out["dW"]))


def _worker(rank, world, port, agg, fail_rank, q):
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    import torch.distributed as dist
    try:
        dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world,
                                timeout=datetime.timedelta(seconds=5))
        w, H, W, y, m, old, ref, adv = _batch()
        resp, rows = dp.shard_rows(w.n_prompts, w.G, w.L, world, rank)
        n_local = resp.stop - resp.start
        local = float(m[rows].sum()) if agg == 0 else float(n_local)
        if rank == fail_rank:
            raise RuntimeError("planted failure before the collective")
        loss, dH, dW = dp.dp_loss_fwd_bwd(H[rows], W, y[rows], m[rows], old[rows], ref[rows], adv[resp],
                                          n_local, w.L, w.clip_eps, w.beta, agg, local,
                                          compute=_oracle_compute)
        q.put((rank, "ok", float(loss.item()), dH.numpy(), dW.numpy(), rows.start, rows.stop))
    except Exception:  # reported to the parent, never swallowed
        q.put((rank, "error", traceback.format_exc(), None, None, None, None))
    finally:
        if dist.is_initialized():
            try:
                dist.destroy_process_group()
            except Exception:
                pass


def _run(agg, fail_rank=-1, world=2):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, agg, fail_rank, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = {}
    for _ in range(world):
        item = q.get(timeout=120)
        res[item[0]] = item
    for p in procs:
        p.join(timeout=60)
        if p.is_alive():
            p.kill()
    return res


@pytest.mark.parametrize("agg", [0, 1])
def test_two_ranks_equal_the_whole_batch(agg):
    import oracle
    res = _run(agg)
    for r in range(2):
        assert res[r][1] == "ok", res[r][2]
    w, H, W, y, m, old, ref, adv = _batch()
    full = oracle.loss_fwd_bwd(H, W, y, m, old, ref, adv, w.n_resp, w.L, w.clip_eps, w.beta, agg)
    for r in range(2):
        _, _, loss, dH, dW, a, b = res[r]
        assert loss == pytest.approx(full["loss"], rel=1e-12, abs=1e-15)
        np.testing.assert_allclose(dW, full["dW"], rtol=1e-11, atol=1e-15)
        np.testing.assert_allclose(dH, full["dH"][a:b], rtol=1e-11, atol=1e-15)


def test_failed_rank_makes_the_other_raise_not_hang():
    res = _run(0, fail_rank=1)
    assert res[1][1] == "error" and "planted failure" in res[1][2]
    assert res[0][1] == "error"  # the collective timed out or saw the peer leave


def _bench_worker(rank, world, port, q):
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    import torch.distributed as dist
    try:
        import bench
        dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world,
                                timeout=datetime.timedelta(seconds=20))
        dt, n = bench.across_ranks(torch, torch.device("cpu"), dist, 0.25 + 0.5 * rank, 1000 + 7 * rank)
        q.put((rank, "ok", dt, n))
    except Exception:  # reported to the parent, never swallowed
        q.put((rank, "error", traceback.format_exc(), None))
    finally:
        if dist.is_initialized():
            dist.destroy_process_group()


def test_bench_end_to_end_numbers_combine_slowest_rank_and_all_tokens():
    """The end-to-end figure across ranks is every rank's tokens over the
    slowest rank's time, the same rule as the device-timed value."""
    import bench
    assert bench.across_ranks(torch, torch.device("cpu"), None, 0.5, 10) == (0.5, 10)
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_bench_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = dict((item[0], item) for item in (q.get(timeout=120) for _ in procs))
    for p in procs:
        p.join(timeout=60)
        if p.is_alive():
            p.kill()
    for r in range(2):
        assert res[r][1] == "ok", res[r][2]
        assert res[r][2] == pytest.approx(0.75) and res[r][3] == 2007
