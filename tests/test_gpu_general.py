"""Parity of the general retrieval path (through the C ABI) with the CPU oracle:
one list per layer (head-averaged weights) and retrieval over compressed windows."""
import numpy as np
import pytest
import torch

from oracle import kmeans as KM
from oracle import retrieval as R
from tests import parity as PY

pytestmark = pytest.mark.gpu

# Head-averaged weights carry the relative rounding of the per-head weights they
# average: |dw / w| <= |ds| (natural-log units) + fp32 rounding, with |ds| <= TOL_SCORE.
REL_ALPHA = 1e-3


def _ss():
    import paper_2609_02780_gb300 as ss
    return ss


def _bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


def _keys_q(seed, P, Hq, Hkv, F, Tf, R_rows=4, scene=0):
    g = torch.Generator().manual_seed(seed)
    keys = torch.randn(P, Hkv, F * Tf, 128, generator=g)
    if scene:
        means = 0.7 * torch.randn(P, Hkv, F // scene + 1, 1, 128, generator=g)
        keys += means.repeat_interleave(scene * Tf, 2)[:, :, :F * Tf, 0]
    q = torch.randn(P, R_rows, Hq, 128, generator=g)
    return keys.to(torch.bfloat16), q.to(torch.bfloat16)


def _mean_case(keys, q, *, Tf, fpu, k, budget, n_recent, q_agg=0):
    ss = _ss()
    P, Hkv, N, _ = keys.shape
    Hq = q.shape[2]
    F = N // Tf
    idx = ss.Index(P, Hq, Hkv, Tf, F, frames_per_unit=fpu, device="cuda")
    idx.append(keys.cuda())
    res = idx.retrieve(q.cuda(), k=k, budget=budget, n_recent=n_recent, q_agg=q_agg,
                       head_agg=ss.H_MEAN)
    res.check()
    Tu, U = Tf * fpu, F // fpu
    Uh = max(0, U - n_recent)
    gpu = PY.gpu_outputs(res, Uh)
    kb, qb = _bits(keys), _bits(q)
    desc = R.descriptors(kb, U, Tu)
    ref = R.retrieve(kb, qb, n_units=U, tokens_per_unit=Tu, k=k, budget=budget,
                     frames_per_unit=fpu, n_recent=n_recent, q_agg=q_agg,
                     head_agg=R.H_MEAN, desc=desc)
    assert gpu["topk_tok"].shape[0] == P
    info = PY.check_topk(ref["alpha"], gpu["topk_tok"], gpu["topk_w"], ref["alpha"], k,
                         rel_tol=REL_ALPHA)
    # list statistics of a layer list: (max alpha, sum alpha = 1)
    st = gpu["list_stats"]
    assert np.allclose(st[:, 0], ref["alpha"].max(1), rtol=REL_ALPHA)
    assert np.allclose(st[:, 1], 1.0, atol=1e-4)
    assert np.allclose(gpu["mass"], ref["mass"], rtol=1e-3, atol=1e-7)
    info.update(PY.check_chain(gpu, desc, Uh, Tu, budget, 4, 1, fpu))
    assert gpu["votes"].sum() == P * min(k, Uh * Tu)
    info["e2e"] = PY.check_end_to_end(gpu, ref, info["ambiguous_lists"], desc, budget,
                                      rel_mass=1e-3)
    return gpu, ref, info


def test_head_averaged_lists_paper_configuration():
    # Table 4's setting: 2-frame units, k = 64 per layer, pool 32, K = 8, 6 recent units
    from paper_2609_02780_gb300 import synth
    w = synth.PRESETS["paper_qwen"]
    data = synth.make_workload(w, device="cpu")
    _mean_case(data["keys"], data["q"], Tf=w.tokens_per_frame, fpu=w.frames_per_unit,
               k=w.k, budget=w.budget, n_recent=w.n_recent)


def test_head_averaged_lists_ragged_and_mean_logit_rows():
    keys, q = _keys_q(31, P=2, Hq=8, Hkv=2, F=70, Tf=23, R_rows=5)
    _mean_case(keys, q, Tf=23, fpu=1, k=200, budget=5, n_recent=3, q_agg=1)


def test_head_averaged_lists_more_tokens_than_the_sort_buffer():
    # 40,000 candidates per list: the top-k goes through the histogram fallback
    keys, q = _keys_q(32, P=1, Hq=4, Hkv=1, F=200, Tf=200, R_rows=2)
    _mean_case(keys, q, Tf=200, fpu=1, k=300, budget=6, n_recent=0)


def _cluster_case(keys, q, *, Tf, fpu, WF, n_c, compressions, k, budget, n_recent,
                  iters=3):
    """compressions: (first_frame, n_frames) of each ss_index_compress call, in order."""
    ss = _ss()
    P, Hkv, N, _ = keys.shape
    Hq = q.shape[2]
    F = N // Tf
    idx = ss.Index(P, Hq, Hkv, Tf, F, frames_per_unit=fpu, device="cuda")
    idx.append(keys.cuda())
    for f0, nf in compressions:
        idx.compress(WF, n_centroids=n_c, iters=iters, first_frame=f0, n_frames=nf)
    res = idx.retrieve(q.cuda(), k=k, budget=budget, n_recent=n_recent, use_clusters=1)
    res.check()
    cl = idx.clusters()
    Tu, U = Tf * fpu, F // fpu
    Uh = max(0, U - n_recent)
    gpu = PY.gpu_outputs(res, Uh)
    kb, qb = _bits(keys), _bits(q)
    desc = R.descriptors(kb, U, Tu)
    comp = PY.gpu_comp(cl, Tf, fpu)                          # the GPU's own clusters
    assert comp["window_first_frames"] == [f0 + j * WF for f0, nf in compressions
                                           for j in range(nf // WF)]
    ref = KM.retrieve_compressed(kb, qb, comp, n_units=U, tokens_per_unit=Tu,
                                 frames_per_unit=fpu, tokens_per_frame=Tf, k=k,
                                 budget=budget, n_recent=n_recent, desc=desc)
    info = PY.check_topk(ref["s"], gpu["topk_tok"], gpu["topk_w"], ref["w"], k,
                         ids=ref["ids"])
    PY.check_stats(ref["s"], gpu["list_stats"])
    assert np.allclose(gpu["mass"], ref["mass"], rtol=1e-3, atol=1e-7)
    votes = KM.compressed_votes(gpu["topk_tok"], comp["assign"], n_q_heads=Hq,
                                n_kv_heads=Hkv, n_centroids=n_c, window_frames=WF,
                                window_first=comp["window_first_frames"],
                                tokens_per_frame=Tf, tokens_per_unit=Tu, n_hist_units=Uh)
    info.update(PY.check_chain(gpu, desc, Uh, Tu, budget, 4, 1, fpu, votes=votes))
    # a selected centroid votes once per member token
    sizes = cl["member_sizes"].cpu().numpy()
    expect = 0
    for li in range(P * Hq):
        i, g = li // Hq, (li % Hq) // (Hq // Hkv)
        for v in gpu["topk_tok"][li]:
            if v >= KM.CID_BASE:
                w, c = divmod(int(v) - KM.CID_BASE, n_c)
                expect += int(sizes[i, g, w, c])
            elif v >= 0:
                expect += 1
    assert gpu["votes"].sum() <= expect          # members past the history do not vote
    info["e2e"] = PY.check_end_to_end(gpu, ref, info["ambiguous_lists"], desc, budget,
                                      rel_mass=1e-3)
    return gpu, ref, info


def test_compressed_windows_and_raw_tail():
    # 12 of 20 windows compressed; the raw tail and the recent units stay tokens
    keys, q = _keys_q(33, P=2, Hq=8, Hkv=2, F=80, Tf=30, scene=8)
    gpu, ref, _ = _cluster_case(keys, q, Tf=30, fpu=1, WF=4, n_c=16, compressions=[(0, 48)],
                                k=120, budget=6, n_recent=5)
    assert (gpu["topk_tok"] >= KM.CID_BASE).any() and (
        (gpu["topk_tok"] >= 0) & (gpu["topk_tok"] < KM.CID_BASE)).any()


def test_all_history_compressed_two_frame_units_window_past_history():
    # every window compressed; with 3 recent units the last window straddles the history
    keys, q = _keys_q(34, P=1, Hq=4, Hkv=1, F=48, Tf=20, scene=6)
    _cluster_case(keys, q, Tf=20, fpu=2, WF=4, n_c=10, compressions=[(0, 48)], k=40,
                  budget=4, n_recent=3)


def test_windows_after_frame_zero_with_a_raw_gap():
    # two compressions that start after frame 0 and leave raw frames before, between and
    # after them; centroids span two units unequally; the last window holds recent units
    keys, q = _keys_q(36, P=2, Hq=8, Hkv=2, F=60, Tf=12, scene=5)
    gpu, ref, _ = _cluster_case(keys, q, Tf=12, fpu=1, WF=4, n_c=12,
                                compressions=[(8, 16), (32, 24)], k=90, budget=5,
                                n_recent=6)
    tok = gpu["topk_tok"]
    assert (tok >= KM.CID_BASE).any() and ((tok >= 0) & (tok < KM.CID_BASE)).any()
    # centroid ids of the second compression's windows were selected
    assert (tok >= KM.CID_BASE + 4 * 12).any()


def test_windows_after_frame_zero_two_frame_units():
    keys, q = _keys_q(37, P=1, Hq=4, Hkv=1, F=64, Tf=10, scene=8)
    _cluster_case(keys, q, Tf=10, fpu=2, WF=8, n_c=20, compressions=[(16, 16), (40, 16)],
                  k=60, budget=4, n_recent=2)


def test_general_path_errors():
    ss = _ss()
    keys, q = _keys_q(35, P=1, Hq=4, Hkv=1, F=8, Tf=10)
    idx = ss.Index(1, 4, 1, 10, 8, device="cuda")
    idx.append(keys.cuda())
    with pytest.raises(ss.ShallowStreamError, match="STATE"):
        idx.retrieve(q.cuda(), k=5, budget=2, use_clusters=1)
    idx.compress(4, n_centroids=8, iters=2)
    with pytest.raises(ss.ShallowStreamError, match="UNSUPPORTED"):
        idx.retrieve(q.cuda(), k=5, budget=2, use_clusters=1, head_agg=ss.H_MEAN)


def test_general_path_batched_equals_single():
    # one launch per stage over problems of different lengths and compression states
    ss = _ss()
    for mode in ("mean", "clusters"):
        idxs, qs = [], []
        for j, F in enumerate((40, 64, 24)):
            keys, q = _keys_q(40 + j, P=2, Hq=8, Hkv=2, F=F, Tf=20, scene=4)
            ix = ss.Index(2, 8, 2, 20, F, device="cuda")
            ix.append(keys.cuda())
            if mode == "clusters":
                ix.compress(4, n_centroids=8, iters=2, first_frame=0, n_frames=(F // 2) // 4 * 4)
            idxs.append(ix)
            qs.append(q.cuda())
        p = ss.RetrieveParams(k=30, budget=4, n_recent=1,
                              head_agg=ss.H_MEAN if mode == "mean" else ss.H_PER_QHEAD,
                              use_clusters=1 if mode == "clusters" else 0)
        batched = ss.retrieve_batched(idxs, qs, p)
        for ix, q, rb in zip(idxs, qs, batched):
            rs = ix.retrieve(q, k=p.k, budget=p.budget, n_recent=p.n_recent,
                             head_agg=p.head_agg, use_clusters=p.use_clusters)
            uh = ix.n_units - p.n_recent
            for name in ("topk_tok", "topk_w", "list_stats", "counts"):
                assert torch.equal(getattr(rb, name), getattr(rs, name)), (mode, name)
            assert torch.equal(rb.unit_votes[:uh], rs.unit_votes[:uh]), mode
            assert torch.equal(rb.unit_mass[:uh], rs.unit_mass[:uh]), mode
            assert rb.host() == rs.host(), mode
