"""Parity of the paper's long-history compression (ss_index_cluster_units, Eq. 6-7),
the budget (Eq. 5), the cluster evidence (ss_select_clusters, Eq. 13) and retrieval
over the detailed history with the CPU oracle, through the C ABI.

Cluster decisions compare an fp32 dot product with tau, so the GPU's assignment is
checked step by step: the oracle replays each unit's decision from the GPU's own
clusters (its centroid before the unit) and must agree wherever |k . c - tau| exceeds
1e-5; centroids within 1e-5, representative keys within 1e-5 relative of the fp64
running averages of the GPU's memberships."""
import numpy as np
import pytest
import torch

from oracle import retrieval as R
from oracle import unit_clusters as UC
from tests import parity as PY

pytestmark = pytest.mark.gpu


def _ss():
    import paper_2609_02780_gb300 as ss
    return ss


def _bits(t):
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


def _stream(seed, P=2, Hq=8, Hkv=2, F=60, Tf=24, scene=6, R_rows=3):
    g = torch.Generator().manual_seed(seed)
    keys = torch.randn(P, Hkv, F * Tf, 128, generator=g)
    means = 1.5 * torch.randn(P, Hkv, F // scene + 1, 1, 128, generator=g)
    keys += means.repeat_interleave(scene * Tf, 2)[:, :, :F * Tf, 0]
    q = torch.randn(P, R_rows, Hq, 128, generator=g)
    return keys.to(torch.bfloat16), q.to(torch.bfloat16)


def _check_clusters(kb, desc, Tu, uc, tau):
    """Replay every decision from the GPU's own state; returns the ambiguous count."""
    gpu_assign = uc["unit_cluster"].cpu().numpy().tolist()
    cen = uc["centroids"].cpu().double().numpy()
    sizes = uc["sizes"].cpu().numpy()
    n_cl = len(gpu_assign)
    # rebuild the oracle state from the GPU memberships, checking each decision
    amb = 0
    state = None
    for t in range(n_cl):
        if state is not None and state["centroids"]:
            dot = float(desc[t] @ state["centroids"][-1])
            joined = gpu_assign[t] == len(state["centroids"]) - 1
            if abs(dot - tau) > 1e-5:
                assert joined == (dot >= tau), f"unit {t}: decision differs (dot {dot})"
            else:
                amb += 1
        # follow the GPU's decision
        if state is not None and gpu_assign[t] == len(state["centroids"]) - 1:
            state = UC.cluster_units(desc, kb, Tu, [t], -np.inf, state)      # join
        else:
            state = UC.cluster_units(desc, kb, Tu, [t], np.inf, state)       # new cluster
        assert len(state["centroids"]) - 1 == gpu_assign[t]
    assert np.array_equal(sizes, np.array(state["counts"]))
    assert np.allclose(cen, np.array(state["centroids"]), atol=1e-5)
    reps = uc["keys"].cpu().double().numpy()
    ref = np.array(state["reps"])
    assert np.all(np.abs(reps - ref) <= 1e-5 * np.abs(ref) + 1e-5)
    return amb, state


def test_clustering_in_two_calls_scores_and_detailed_retrieval():
    ss = _ss()
    keys, q = _stream(70)
    P, Hkv, N, _ = keys.shape
    Hq, Tf, F = q.shape[2], 24, N // 24
    idx = ss.Index(P, Hq, Hkv, Tf, F, device="cuda")
    idx.append(keys.cuda())
    tau = 0.55
    unit_bytes = P * Hkv * Tf * 128 * 2
    n = idx.units_over_budget(budget_bytes=25 * unit_bytes, near_term_units=10)
    assert n == F - 25
    idx.cluster_units(20, tau, max_clusters=40)          # two calls: the latest cluster
    idx.cluster_units(n - 20, tau, max_clusters=40)      # continues across them
    uc = idx.unit_clusters()
    assert uc["n_clustered_units"] == n
    kb, qb = _bits(keys), _bits(q)
    desc = R.descriptors(kb, F, Tf)
    amb, state = _check_clusters(kb, desc, Tf, uc, tau)
    assert len(state["centroids"]) > 3
    # cluster evidence (Eq. 13)
    for q_agg in (0, 1):
        sel = idx.select_clusters(q.cuda(), k_l=4, q_agg=q_agg)
        torch.cuda.synchronize()
        sc_ref = UC.cluster_scores(qb, np.array(state["centroids"]), Hkv, q_agg)
        got = sel["ids"].cpu().numpy()
        m = int(sel["count"].item())
        assert m == min(4, len(sc_ref))
        assert np.allclose(sel["scores"].cpu().numpy()[:m], sc_ref[got[:m]], atol=1e-5)
        theta = np.sort(sc_ref)[::-1][m - 1]
        assert (sc_ref[got[:m]] >= theta - 1e-5).all()
        assert set(np.nonzero(sc_ref > theta + 1e-5)[0]) <= set(got[:m].tolist())
    # retrieval over the detailed history [n, U - N_r)
    res = idx.retrieve(q.cuda(), k=60, budget=4, n_recent=3)
    res.check()
    Uh = F - 3
    gpu = PY.gpu_outputs(res, Uh)
    ref = UC.retrieve_detailed(kb, qb, n, n_units=F, tokens_per_unit=Tf, k=60, budget=4,
                               n_recent=3, desc=desc)
    ref_full_s = R.scores(R.query_effective(qb), kb[:, :, n * Tf:], (Uh - n) * Tf)
    # the token lists in stream numbering
    tok_local = np.where(gpu["topk_tok"] >= 0, gpu["topk_tok"] - n * Tf, -1)
    info = PY.check_topk(ref_full_s, tok_local, gpu["topk_w"], R.softmax(ref_full_s), 60)
    assert (gpu["votes"][:n] == 0).all() and (gpu["mass"][:n] == 0).all()
    assert np.allclose(gpu["mass"][n:], ref["mass"][n:], rtol=1e-4, atol=1e-7)
    assert gpu["votes"].sum() == P * Hq * 60
    assert (gpu["pool"] >= n).all() and (gpu["sel"] >= n).all() and (gpu["expanded"] >= n).all()
    print("detailed retrieval:", PY.check_end_to_end(gpu, ref, info["ambiguous_lists"], desc, 4))


def test_tau_extremes_and_errors():
    ss = _ss()
    keys, q = _stream(71, F=20)
    P, Hkv, N, _ = keys.shape
    Hq, Tf, F = q.shape[2], 24, 20
    kb = _bits(keys)
    desc = R.descriptors(kb, F, Tf)
    for tau, expect in ((2.0, list(range(12))), (-2.0, [0] * 12)):
        idx = ss.Index(P, Hq, Hkv, Tf, F, device="cuda")
        idx.append(keys.cuda())
        idx.cluster_units(12, tau, max_clusters=12)
        uc = idx.unit_clusters()
        assert uc["unit_cluster"].cpu().tolist() == expect
        _check_clusters(kb, desc, Tf, uc, tau)
    with pytest.raises(ss.ShallowStreamError, match="INVALID_ARG"):
        idx.cluster_units(100, 0.5, max_clusters=12)                  # beyond the units
    with pytest.raises(ss.ShallowStreamError, match="INVALID_ARG"):
        idx.cluster_units(1, 0.5, max_clusters=13)                    # another capacity
    with pytest.raises(ss.ShallowStreamError, match="STATE"):
        idx.compress(4, n_centroids=8, iters=2, first_frame=12, n_frames=8)
    fresh = ss.Index(P, Hq, Hkv, Tf, F, device="cuda")
    fresh.append(keys.cuda())
    with pytest.raises(ss.ShallowStreamError, match="STATE"):
        fresh.select_clusters(q.cuda(), k_l=2)
