"""Retrieval over an index split by token range, with the shards on one GPU: each shard
is its own index over its unit range (ss_retrieve_shard), the payloads are brought to
the host and merged (ss_merge_shards). The merged per-list top-k must equal the
single-index retrieval's exactly (the same kernels score every token the same way, and
each shard's top-k is exact); weights, statistics and mass agree to rounding; votes
exactly; selection and frames equal where no decision is inside its band, and against
the CPU oracle as for any retrieval."""
import numpy as np
import pytest
import torch

from oracle import retrieval as R
from tests import parity as PY

pytestmark = pytest.mark.gpu


def _ss():
    import paper_2609_02780_gb300 as ss
    return ss


def _sharded(keys, q, w_frames_per_unit, Tf, bounds, p):
    """keys bf16 [P][Hkv][F*Tf][d] on the GPU; bounds in units; returns the merged result
    and the payloads."""
    ss = _ss()
    P, Hkv = keys.shape[0], keys.shape[1]
    Hq = q.shape[2]
    fpu = w_frames_per_unit
    Tu = Tf * fpu
    payloads = []
    for i in range(len(bounds) - 1):
        u0, u1 = bounds[i], bounds[i + 1]
        idx = ss.Index(P, Hq, Hkv, Tf, (u1 - u0) * fpu, frames_per_unit=fpu, device=keys.device)
        idx.append(keys[:, :, u0 * Tu:u1 * Tu].contiguous())
        last = i == len(bounds) - 2
        ps = ss.RetrieveParams(k=p.k, budget=p.budget, pool_mult=p.pool_mult, n_prev=p.n_prev,
                               n_recent=p.n_recent if last else 0, q_agg=p.q_agg)
        out = idx.retrieve_shard(q, ps, u0)
        torch.cuda.synchronize()
        assert int(out["status"].item()) == 0
        payloads.append({k: (v.cpu().numpy() if isinstance(v, torch.Tensor) else v)
                         for k, v in out.items() if k != "_keep" and k != "status"})
        payloads[-1]["desc"] = idx.descriptors()[:out["n_units"]].cpu().numpy()
        del idx
    merged = ss.merge_shards(payloads, P * Hq, Tu, p, frames_per_unit=fpu)
    return merged, payloads


def _single(keys, q, Tf, fpu, p):
    ss = _ss()
    P, Hkv = keys.shape[0], keys.shape[1]
    F = keys.shape[2] // Tf
    idx = ss.Index(P, q.shape[2], Hkv, Tf, F, frames_per_unit=fpu, device=keys.device)
    idx.append(keys)
    res = idx.retrieve(q, k=p.k, budget=p.budget, pool_mult=p.pool_mult, n_prev=p.n_prev,
                       n_recent=p.n_recent, q_agg=p.q_agg)
    res.check()
    return idx, res


def _against_single(merged, res, Uh, rel_mass):
    tok = res.topk_tok.cpu().numpy()
    assert np.array_equal(merged["topk_tok"], tok), "merged top-k differs from one index"
    assert np.allclose(merged["topk_w"], res.topk_w.cpu().numpy(), rtol=1e-5, atol=1e-12)
    st = res.list_stats.cpu().numpy()
    assert np.allclose(merged["list_stats"][:, 0], st[:, 0], atol=0)
    assert np.allclose(merged["list_stats"][:, 1], st[:, 1], rtol=1e-5)
    assert np.array_equal(merged["votes"], res.unit_votes[:Uh].cpu().numpy())
    assert np.allclose(merged["mass"], res.unit_mass[:Uh].cpu().numpy(), rtol=rel_mass, atol=1e-9)


def test_three_shards_small_stream():
    ss = _ss()
    g = torch.Generator().manual_seed(50)
    P, Hq, Hkv, F, Tf = 2, 8, 2, 60, 30
    keys = (torch.randn(P, Hkv, F * Tf, 128, generator=g) +
            0.5 * torch.randn(P, Hkv, F // 6, 1, 128, generator=g).repeat_interleave(6 * Tf, 2)
            .view(P, Hkv, F * Tf, 128)).to(torch.bfloat16)
    q = torch.randn(P, 4, Hq, 128, generator=g).to(torch.bfloat16)
    p = ss.RetrieveParams(k=200, budget=6, n_recent=4)
    kd, qd = keys.cuda(), q.cuda()
    merged, _ = _sharded(kd, qd, 1, Tf, [0, 17, 41, 60], p)
    idx, res = _single(kd, qd, Tf, 1, p)
    Uh = F - p.n_recent
    _against_single(merged, res, Uh, 1e-4)
    # and the oracle
    kb = keys.view(torch.int16).numpy().view(np.uint16)
    qb = q.view(torch.int16).numpy().view(np.uint16)
    ref = R.retrieve(kb, qb, n_units=F, tokens_per_unit=Tf, k=p.k, budget=p.budget,
                     n_recent=p.n_recent)
    info = PY.check_topk(ref["s"], merged["topk_tok"], merged["topk_w"], ref["w"], p.k)
    desc = R.descriptors(kb, F, Tf)
    g_like = {k: np.asarray(v).astype(np.int64) if k != "mass" else v for k, v in merged.items()}
    g_like["mass"] = merged["mass"]
    PY.check_chain(g_like, desc, Uh, Tf, p.budget, 4, 1, 1)
    print("three shards:", PY.check_end_to_end(g_like, ref, info["ambiguous_lists"], desc, p.budget))


def test_one_hour_index_in_four_shards():
    ss = _ss()
    from paper_2609_02780_gb300 import synth
    w = synth.PRESETS["hour1"]
    data = synth.make_workload(w, device=torch.device("cuda"))
    p = ss.RetrieveParams(k=w.k, budget=w.budget, pool_mult=w.pool_mult, n_prev=w.n_prev,
                          n_recent=w.n_recent, q_agg=w.q_agg)
    merged, _ = _sharded(data["keys"], data["q"], w.frames_per_unit, w.tokens_per_frame,
                         [0, 900, 1800, 2700, 3600], p)
    idx, res = _single(data["keys"], data["q"], w.tokens_per_frame, w.frames_per_unit, p)
    Uh = w.n_hist_units
    _against_single(merged, res, Uh, 1e-4)
    single = res.host()
    # the merge's own pool, max-min and expansion follow the rules from its votes and mass
    desc = idx.descriptors().cpu().double().numpy()
    g_like = {k: np.asarray(v).astype(np.int64) for k, v in merged.items()
              if k in ("topk_tok", "votes", "pool", "sel", "expanded", "frames")}
    g_like["mass"] = merged["mass"]
    PY.check_chain(g_like, desc, Uh, w.tokens_per_unit, w.budget, w.pool_mult, w.n_prev,
                   w.frames_per_unit)
    # the selection: equal to one index's unless a pool or greedy decision is within rounding
    same = merged["frames"].tolist() == single["frames"]
    print("hour1 in four shards: frames", "equal to one index" if same else "differ")
