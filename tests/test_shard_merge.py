"""Retrieval over an index split by token range (one shard per GPU), on CPU ranks:

* each shard's payload comes from the oracle (oracle/shard.py): its own top-k tokens with
  scores, its list and per-unit softmax statistics, its descriptors;
* the library's host merge (ss_merge_shards, through the C ABI; no GPU) combines them;
* the merged lists, weights, votes, mass, pool, selection and frames must be the
  unsharded oracle retrieval's (banded where fp32 scores may reorder near-ties).

The multi-rank tests run the shards as gloo ranks (world size 2 and 4): every rank
computes its payload, one gather brings them to rank 0, rank 0 merges.
"""
import os
import socket

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

from oracle import retrieval as R
from oracle import shard as SH
from tests import parity as PY

P_, HQ, HKV, TU, U, K, BUDGET = 2, 8, 2, 20, 30, 50, 4


def to_bits(t: torch.Tensor) -> np.ndarray:
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


def _data(seed=0):
    g = torch.Generator().manual_seed(seed)
    keys = torch.randn(P_, HKV, U * TU, 128, generator=g)
    scene = 0.6 * torch.randn(P_, HKV, U // 5 + 1, 128, generator=g)
    keys += scene.repeat_interleave(5 * TU, 2)[:, :, :U * TU]
    q = torch.randn(P_, 3, HQ, 128, generator=g)
    return to_bits(keys.to(torch.bfloat16)), to_bits(q.to(torch.bfloat16))


def _payloads(kb, qb, bounds, n_recent):
    """Shards over units [bounds[i], bounds[i + 1]); the last one holds the recent units."""
    out = []
    for i in range(len(bounds) - 1):
        u0, u1 = bounds[i], bounds[i + 1]
        last = i == len(bounds) - 2
        n_hist = (u1 - u0) - (n_recent if last else 0)
        out.append(SH.shard_payload(kb[:, :, u0 * TU:u1 * TU], qb, unit_begin=u0,
                                    n_units=n_hist, tokens_per_unit=TU, k=K))
    return out


def _merge(payloads, n_recent=0):
    import paper_2609_02780_gb300 as ss
    p = ss.RetrieveParams(k=K, budget=BUDGET, n_recent=n_recent)
    return ss.merge_shards(payloads, P_ * HQ, TU, p)


def _compare(merged, kb, qb, n_recent):
    ref = R.retrieve(kb, qb, n_units=U, tokens_per_unit=TU, k=K, budget=BUDGET, n_recent=n_recent)
    Uh = U - n_recent
    info = PY.check_topk(ref["s"], merged["topk_tok"], merged["topk_w"], ref["w"], K)
    st = merged["list_stats"]
    PY.check_stats(ref["s"], st)
    assert len(merged["votes"]) == Uh
    assert np.allclose(merged["mass"], ref["mass"], rtol=1e-5, atol=1e-9)
    gpu_like = {"topk_tok": merged["topk_tok"], "votes": merged["votes"].astype(np.int64),
                "mass": merged["mass"], "pool": merged["pool"].astype(np.int64),
                "sel": merged["sel"].astype(np.int64), "expanded": merged["expanded"].astype(np.int64),
                "frames": merged["frames"].astype(np.int64)}
    desc = R.descriptors(kb, U, TU)
    info.update(PY.check_chain(gpu_like, desc, Uh, TU, BUDGET, 4, 1, 1))
    e2e = PY.check_end_to_end(gpu_like, ref, info["ambiguous_lists"], desc, BUDGET)
    return info, e2e


@pytest.mark.parametrize("bounds,n_recent", [([0, 13, 30], 0), ([0, 7, 8, 21, 30], 3),
                                              ([0, 2, 30], 5)])
def test_merged_shards_equal_the_unsharded_retrieval(bounds, n_recent):
    kb, qb = _data(1)
    merged = _merge(_payloads(kb, qb, bounds, n_recent), n_recent)
    info, e2e = _compare(merged, kb, qb, n_recent)
    assert info["ambiguous_lists"] == 0 and e2e == "e2e ids exact", (info, e2e)


def test_shard_with_fewer_tokens_than_k():
    # a one-unit shard holds 20 tokens < k = 50: its whole history is its candidate list
    kb, qb = _data(2)
    merged = _merge(_payloads(kb, qb, [0, 1, 30], 0))
    _, e2e = _compare(merged, kb, qb, 0)
    assert e2e == "e2e ids exact"


def test_merge_rejects_shards_that_do_not_tile_the_history():
    import paper_2609_02780_gb300 as ss
    kb, qb = _data(3)
    pl = _payloads(kb, qb, [0, 10, 30], 0)
    pl[1] = dict(pl[1], unit_begin=11)
    with pytest.raises(ss.ShallowStreamError, match="INVALID_ARG"):
        _merge(pl)
    pl = _payloads(kb, qb, [0, 10, 30], 0)
    with pytest.raises(ss.ShallowStreamError, match="UNSUPPORTED"):
        ss.merge_shards(pl, P_ * HQ, TU, ss.RetrieveParams(k=K, budget=BUDGET, head_agg=ss.H_MEAN))


# ---------------------------------------------------------------- gloo ranks
def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, bounds, n_recent, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    kb, qb = _data(4)                               # every rank draws the same stream
    u0, u1 = bounds[rank], bounds[rank + 1]
    last = rank == world - 1
    mine = SH.shard_payload(kb[:, :, u0 * TU:u1 * TU], qb, unit_begin=u0,
                            n_units=(u1 - u0) - (n_recent if last else 0),
                            tokens_per_unit=TU, k=K)
    gathered = [None] * world if rank == 0 else None
    dist.gather_object(mine, gathered, dst=0)        # the one exchange step
    if rank == 0:
        merged = _merge(gathered, n_recent)
        info, e2e = _compare(merged, kb, qb, n_recent)
        out.put((info["ambiguous_lists"], e2e, merged["frames"].tolist()))
    dist.destroy_process_group()


@pytest.mark.parametrize("world,bounds,n_recent", [(2, [0, 16, 30], 2), (4, [0, 5, 12, 20, 30], 0)])
def test_gloo_ranks_shard_gather_and_merge(world, bounds, n_recent):
    port = _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, bounds, n_recent, q))
             for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(180)
        assert p.exitcode == 0
    amb, e2e, frames = q.get(timeout=5)
    assert amb == 0 and e2e == "e2e ids exact"
    kb, qb = _data(4)
    ref = R.retrieve(kb, qb, n_units=U, tokens_per_unit=TU, k=K, budget=BUDGET, n_recent=n_recent)
    assert frames == ref["frames"].tolist()
