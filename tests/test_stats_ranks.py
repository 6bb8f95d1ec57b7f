"""The standardisation update under data parallelism, on CPU with two gloo
ranks: each rank adds the moment sums of its own shard and sampled rows, the
sums are added across ranks (``dpb.ema_step``'s all-reduce) and both ranks
then make the same EMA step. The result must equal one process's step over
the whole batch (the sums are linear in the rows), and the ranks' tables must
be identical. The sums and the step come from the oracle here (no GPU): what
is under test is the exchange around them."""
import os
import socket

import numpy as np
import torch
import torch.multiprocessing as mp

import oracle
from paper_2607_20652_gb300 import dpb, inputs

CFG = dict(d=64, m_bits=12, levels=3, children=16, beam=4, k=8)
ALPHA = 0.2


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _shard(rank):
    x = inputs.gaussian_rows(30 + 7 * rank, CFG["d"], 100 + rank).astype(np.float64)
    rows = inputs.sample_rows(len(x), 5, 200 + rank)
    return x, rows


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    cfg = oracle.resolve(**CFG)
    m = 1 << cfg.m_bits
    mu, sigma = inputs.moment_tables(m, 7)
    tables = {"mu": mu.astype(np.float64), "sigma": sigma.astype(np.float64)}
    x, rows = _shard(rank)
    acc = torch.zeros((3, m), dtype=torch.float64)

    def accumulate(a):
        oracle.stats_accumulate(cfg, x, rows, mu=tables["mu"], sigma=tables["sigma"], acc=a.numpy())

    def update(a):
        tables["mu"], tables["sigma"] = oracle.stats_update(a.numpy(), ALPHA, tables["mu"], tables["sigma"])

    dpb.ema_step(accumulate, update, acc)
    q.put((rank, tables["mu"], tables["sigma"], bool(acc.any())))
    dist.destroy_process_group()


def test_two_ranks_step_like_one_process_over_the_whole_batch():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted((q.get(timeout=120) for _ in range(2)), key=lambda o: o[0])
    for p in procs:
        p.join(60)
        assert p.exitcode == 0
    (_, mu0, sg0, left0), (_, mu1, sg1, left1) = out
    assert not left0 and not left1                       # the step consumed the sums
    assert np.array_equal(mu0, mu1) and np.array_equal(sg0, sg1)

    cfg = oracle.resolve(**CFG)
    m = 1 << cfg.m_bits
    mu, sigma = inputs.moment_tables(m, 7)
    (x0, r0), (x1, r1) = _shard(0), _shard(1)
    x = np.concatenate([x0, x1])
    rows = np.concatenate([r0, r1 + len(x0)])
    acc = oracle.stats_accumulate(cfg, x, rows, mu=mu.astype(np.float64), sigma=sigma.astype(np.float64))
    mu_w, sg_w = oracle.stats_update(acc, ALPHA, mu.astype(np.float64), sigma.astype(np.float64))
    assert np.allclose(mu0, mu_w, rtol=0, atol=1e-12) and np.allclose(sg0, sg_w, rtol=0, atol=1e-12)
    assert np.sum(mu_w != mu.astype(np.float64)) > cfg.d      # level 0 and sampled children moved


def test_single_process_skips_the_exchange():
    calls = []
    acc = torch.zeros(3)
    dpb.ema_step(lambda a: calls.append("acc"), lambda a: calls.append("upd"), acc)
    assert calls == ["acc", "upd"]
