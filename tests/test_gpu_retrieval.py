"""Parity of the CUDA retrieval path (through the C ABI) with the CPU oracle."""
import math

import numpy as np
import pytest
import torch

from oracle import retrieval as R
from tests import parity as PY

pytestmark = pytest.mark.gpu


def _ss():
    import paper_2609_02780_gb300 as ss
    return ss


def to_bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


def run_case(keys, q, *, tokens_per_frame, k, budget, frames_per_unit=1, pool_mult=4,
             n_prev=1, n_recent=0, q_agg=0, check_e2e=True, append_chunks=None):
    """Builds an index from keys [P][Hkv][F*T_f][d], retrieves, checks against the oracle."""
    ss = _ss()
    dev = torch.device("cuda")
    P, Hkv, N, d = keys.shape
    Hq = q.shape[2]
    F = N // tokens_per_frame
    idx = ss.Index(P, Hq, Hkv, tokens_per_frame, F, frames_per_unit=frames_per_unit,
                   device=dev)
    kd = keys.to(dev)
    if append_chunks:
        f0 = 0
        for nf in append_chunks:
            idx.append(kd[:, :, f0 * tokens_per_frame:], n_frames=nf)
            f0 += nf
        assert f0 == F
    else:
        idx.append(kd)
    res = idx.retrieve(q.to(dev), k=k, budget=budget, pool_mult=pool_mult, n_prev=n_prev,
                       n_recent=n_recent, q_agg=q_agg)
    res.check()
    Tu = tokens_per_frame * frames_per_unit
    U = F // frames_per_unit
    Uh = max(0, U - n_recent)
    gpu = PY.gpu_outputs(res, Uh)
    kb, qb = to_bits(keys), to_bits(q)
    desc = R.descriptors(kb, U, Tu)
    desc_gpu = idx.descriptors().cpu().double().numpy()
    assert np.abs(desc_gpu - desc).max() <= 1e-5
    ref = R.retrieve(kb, qb, n_units=U, tokens_per_unit=Tu, k=k, budget=budget,
                     frames_per_unit=frames_per_unit, pool_mult=pool_mult, n_prev=n_prev,
                     n_recent=n_recent, q_agg=q_agg, desc=desc)
    info = {}
    if Uh > 0:
        info.update(PY.check_topk(ref["s"], gpu["topk_tok"], gpu["topk_w"], ref["w"], k))
        PY.check_stats(ref["s"], gpu["list_stats"])
        assert np.allclose(gpu["mass"], ref["mass"], rtol=1e-4, atol=1e-6)
    else:
        assert (gpu["topk_tok"] == -1).all()
    info.update(PY.check_chain(gpu, desc, Uh, Tu, budget, pool_mult, n_prev, frames_per_unit))
    n_valid = (gpu["topk_tok"] >= 0).sum()
    assert gpu["votes"].sum() == n_valid == P * Hq * min(k, Uh * Tu)
    if check_e2e and Uh > 0:
        info["e2e"] = PY.check_end_to_end(gpu, ref, info.get("ambiguous_lists", 0), desc,
                                          budget, pool_mult)
    return idx, res, gpu, ref, info


def gaussian_case(seed, P, Hq, Hkv, F, Tf, R_rows=4, planted=(), scale=1.0):
    g = torch.Generator().manual_seed(seed)
    keys = torch.randn(P, Hkv, F * Tf, 128, generator=g) * scale
    q = torch.randn(P, R_rows, Hq, 128, generator=g)
    G = Hq // Hkv
    for f in planted:
        for i in range(P):
            for j in range(Hkv):
                keys[i, j, f * Tf:(f + 1) * Tf] += 0.5 * q[i, -1, j * G:(j + 1) * G].mean(0)
    return keys.to(torch.bfloat16), q.to(torch.bfloat16)


def test_tiny_preset_parity():
    from paper_2609_02780_gb300 import synth
    w = synth.PRESETS["tiny"]
    data = synth.make_workload(w, device="cpu")
    _, _, gpu, ref, info = run_case(data["keys"], data["q"], tokens_per_frame=w.tokens_per_frame,
                                    k=w.k, budget=w.budget)
    # the planted frames carry the question's direction: all of them lead the pool
    assert set(data["planted"]) <= set(gpu["pool"][:8].tolist())


def test_ragged_units_many_chunks():
    # 196-token frames end in a partial 16-row tile; 300 units split over many CTAs
    keys, q = gaussian_case(1, P=2, Hq=28, Hkv=4, F=300, Tf=196, R_rows=8, planted=(7, 150, 299))
    run_case(keys, q, tokens_per_frame=196, k=512, budget=16)


def test_mean_logit_rows_and_recent_units():
    keys, q = gaussian_case(2, P=2, Hq=8, Hkv=2, F=120, Tf=36, R_rows=5)
    run_case(keys, q, tokens_per_frame=36, k=100, budget=6, q_agg=1, n_recent=7)


def test_group_sizes_one_and_eight():
    keys, q = gaussian_case(3, P=1, Hq=4, Hkv=4, F=40, Tf=20)
    run_case(keys, q, tokens_per_frame=20, k=33, budget=5)
    keys, q = gaussian_case(4, P=2, Hq=16, Hkv=2, F=40, Tf=20)
    run_case(keys, q, tokens_per_frame=20, k=33, budget=5)


def test_tiny_units_fewer_rows_than_a_tile_and_two_frame_units():
    keys, q = gaussian_case(5, P=2, Hq=8, Hkv=2, F=60, Tf=3)
    run_case(keys, q, tokens_per_frame=3, k=17, budget=4, frames_per_unit=2, n_prev=2)


def test_k_at_least_all_tokens():
    keys, q = gaussian_case(6, P=1, Hq=7, Hkv=1, F=10, Tf=12)
    _, _, gpu, _, _ = run_case(keys, q, tokens_per_frame=12, k=4096, budget=3)
    assert gpu["votes"].tolist() == [7 * 12] * 10


def test_all_scores_equal_lowest_ids_win():
    keys = torch.zeros(1, 2, 30 * 16, 128, dtype=torch.bfloat16)
    q = torch.randn(1, 1, 4, 128).to(torch.bfloat16)
    _, _, gpu, _, _ = run_case(keys, q, tokens_per_frame=16, k=40, budget=3)
    for li in range(4):
        assert gpu["topk_tok"][li].tolist() == list(range(40))


def test_pool_smaller_than_pool_mult_budget_and_empty_history():
    keys, q = gaussian_case(7, P=1, Hq=4, Hkv=2, F=6, Tf=10)
    run_case(keys, q, tokens_per_frame=10, k=8, budget=4)            # pool = 6 units
    _, _, gpu, _, _ = run_case(keys, q, tokens_per_frame=10, k=8, budget=4, n_recent=6)
    assert gpu["counts"] == [0, 0, 0, 0]


def test_incremental_and_strided_appends():
    keys, q = gaussian_case(8, P=2, Hq=8, Hkv=2, F=50, Tf=24)
    run_case(keys, q, tokens_per_frame=24, k=64, budget=5, append_chunks=[1, 13, 20, 16])


def test_deterministic_bitwise():
    ss = _ss()
    keys, q = gaussian_case(9, P=2, Hq=28, Hkv=4, F=200, Tf=49)
    idx = ss.Index(2, 28, 4, 49, 200, device="cuda")
    idx.append(keys.cuda())
    qd = q.cuda()
    first = None
    for _ in range(10):
        r = idx.retrieve(qd, k=300, budget=12)
        out = (r.topk_tok.clone(), r.topk_w.clone(), r.unit_mass.clone(), r.sel_units.clone(),
               r.list_stats.clone())
        if first is None:
            first = out
        else:
            for a, b in zip(first, out):
                assert torch.equal(a, b)


def test_batched_equals_single():
    ss = _ss()
    cases = [gaussian_case(10 + j, P=2, Hq=8, Hkv=2, F=F, Tf=30) for j, F in
             enumerate((40, 90, 17))]
    idxs = []
    for keys, _ in cases:
        ix = ss.Index(2, 8, 2, 30, keys.shape[2] // 30, device="cuda")
        ix.append(keys.cuda())
        idxs.append(ix)
    qs = [q.cuda() for _, q in cases]
    p = ss.RetrieveParams(k=50, budget=4)
    batched = ss.retrieve_batched(idxs, qs, p)
    for ix, q, rb in zip(idxs, qs, batched):
        rs = ix.retrieve(q, k=50, budget=4)
        # softmax sums are combined per unit and then in unit order, whatever CTA scored
        # a unit, so batching changes no bit
        for name in ("topk_tok", "counts", "unit_votes", "topk_w", "list_stats"):
            assert torch.equal(getattr(rb, name), getattr(rs, name)), name
        assert rb.host() == rs.host()


def test_host_entry_point_matches_device_path():
    ss = _ss()
    keys, q = gaussian_case(11, P=2, Hq=8, Hkv=2, F=64, Tf=32)
    idx = ss.Index(2, 8, 2, 32, 64, device="cuda")
    idx.append(keys.cuda())
    p = ss.RetrieveParams(k=70, budget=6)
    host = idx.retrieve_host(q, p)
    dev = idx.retrieve(q.cuda(), k=70, budget=6).host()
    assert host["sel"] == dev["sel"] and host["frames"] == dev["frames"]
    # repeated calls with other questions (the host call copies only the rows it reads
    # under LAST, every row under MEAN_LOGIT) agree with the device path each time
    _, q2 = gaussian_case(12, P=2, Hq=8, Hkv=2, F=64, Tf=32)
    # page-locked rows are read by the kernels in place, pageable rows are copied first;
    # both agree with the device path, under every row reading
    for q_agg in (0, 1, 2):
        pq = ss.RetrieveParams(k=70, budget=6, q_agg=q_agg)
        for qq in (q2, q.pin_memory(), q2.pin_memory(), q):
            host = idx.retrieve_host(qq, pq)
            dev = idx.retrieve(qq.cuda(), k=70, budget=6, q_agg=q_agg).host()
            assert host["sel"] == dev["sel"] and host["frames"] == dev["frames"]
            assert host["expanded"] == dev["expanded"]
            assert host["counts"][1:] == [len(dev["sel"]), len(dev["expanded"]),
                                          len(dev["frames"])]


def test_invalid_arguments_fail_before_launch():
    ss = _ss()
    idx = ss.Index(1, 4, 2, 8, 10, device="cuda")
    with pytest.raises(ss.ShallowStreamError, match="CAPACITY"):
        idx.append(torch.zeros(1, 2, 11 * 8, 128, dtype=torch.bfloat16, device="cuda"))
    idx.append(torch.zeros(1, 2, 10 * 8, 128, dtype=torch.bfloat16, device="cuda"))
    q = torch.zeros(1, 1, 4, 128, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(ss.ShallowStreamError, match="UNSUPPORTED"):
        idx.retrieve(q, k=5000, budget=2)
    with pytest.raises(ss.ShallowStreamError, match="INVALID_ARG"):
        idx.retrieve(q, k=5, budget=0)
    with pytest.raises(ss.ShallowStreamError, match="UNSUPPORTED"):
        ss.Index(1, 4, 2, 8, 10, head_dim=64, device="cuda")


def test_maxmin_pool_sizes_across_the_gram_storage_forms():
    # the Gram triangle of the pool is held in fp32 (pool <= 320), 24-bit fixed point
    # (320 < pool <= 384) or global memory (larger); each must give a valid greedy
    keys, q = gaussian_case(12, P=1, Hq=4, Hkv=1, F=420, Tf=8, R_rows=2)
    for budget in (80, 96, 105):              # pools 320, 384, 420
        run_case(keys, q, tokens_per_frame=8, k=64, budget=budget, check_e2e=False)


def test_maxmin_pool_sizes_that_leave_lanes_past_the_pool():
    # pools that are not a multiple of the greedy's ranks per warp: the lanes' ranks past
    # the pool read past the end of the triangle (fp32 in shared memory: 36 and 260,
    # fixed point: 324, global memory: 516) and must not change the selection
    keys, q = gaussian_case(13, P=1, Hq=4, Hkv=1, F=600, Tf=8, R_rows=2)
    for budget in (9, 65, 81, 129):           # pools 36, 260, 324, 516
        run_case(keys, q, tokens_per_frame=8, k=64, budget=budget, check_e2e=False)
