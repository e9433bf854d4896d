"""Parity of the lists ranked by the mean of the question rows' softmax weights
(SS_Q_MEAN_SOFTMAX; two tcgen05 passes over the keys) with the CPU oracle, through the
C ABI: row-averaged weights of the listed tokens, the per-list top-k band (relative,
as for any averaged weight), list statistics (max weight, weights summing to 1), the
attention mass, and chained votes, pool, max-min and expansion; end to end where no
decision is inside its band. Row counts cover one 16-row group per head (with padding
rows), two MMA row blocks, and the 64-row case whose rows fill two operand tiles."""
import numpy as np
import pytest
import torch

from oracle import retrieval as R
from tests import parity as PY

pytestmark = pytest.mark.gpu

REL_ALPHA = 1e-3


def _ss():
    import paper_2609_02780_gb300 as ss
    return ss


def _bits(t):
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


def _case(seed, P, Hq, Hkv, F, Tf, R_rows, k, budget, n_recent=0, scene=4):
    ss = _ss()
    g = torch.Generator().manual_seed(seed)
    keys = torch.randn(P, Hkv, F * Tf, 128, generator=g)
    means = 0.6 * torch.randn(P, Hkv, F // scene + 1, 1, 128, generator=g)
    keys += means.repeat_interleave(scene * Tf, 2)[:, :, :F * Tf, 0]
    keys = keys.to(torch.bfloat16)
    q = torch.randn(P, R_rows, Hq, 128, generator=g).to(torch.bfloat16)
    idx = ss.Index(P, Hq, Hkv, Tf, F, device="cuda")
    idx.append(keys.cuda())
    res = idx.retrieve(q.cuda(), k=k, budget=budget, n_recent=n_recent, q_agg=ss.Q_MEAN_SOFTMAX)
    res.check()
    U = F
    Uh = U - n_recent
    gpu = PY.gpu_outputs(res, Uh)
    kb, qb = _bits(keys), _bits(q)
    desc = R.descriptors(kb, U, Tf)
    ref = R.retrieve(kb, qb, n_units=U, tokens_per_unit=Tf, k=k, budget=budget,
                     n_recent=n_recent, q_agg=R.Q_MEAN_SOFTMAX, desc=desc)
    info = PY.check_topk(ref["alpha"], gpu["topk_tok"], gpu["topk_w"], ref["alpha"], k,
                         rel_tol=REL_ALPHA)
    st = gpu["list_stats"]
    assert np.allclose(st[:, 0], ref["alpha"].max(1), rtol=REL_ALPHA)
    assert np.allclose(st[:, 1], 1.0, atol=1e-4)
    assert np.allclose(gpu["mass"], ref["mass"], rtol=1e-3, atol=1e-7)
    info.update(PY.check_chain(gpu, desc, Uh, Tf, budget, 4, 1, 1))
    assert gpu["votes"].sum() == P * Hq * min(k, Uh * Tf)
    info["e2e"] = PY.check_end_to_end(gpu, ref, info["ambiguous_lists"], desc, budget,
                                      rel_mass=1e-3)
    return gpu, ref, info


def test_rows_padded_to_sixteen_and_recent_units():
    # 5 rows per head (padded to 16): 7 heads x 16 = 112 operand rows, one MMA row block
    _case(60, P=2, Hq=28, Hkv=4, F=50, Tf=37, R_rows=5, k=120, budget=5, n_recent=3)


def test_thirty_two_rows_two_row_blocks_ragged_tiles():
    # the 1-hour configuration's rows (R = 32, G = 7: 224 rows), 196-token units
    _case(61, P=1, Hq=28, Hkv=4, F=40, Tf=196, R_rows=32, k=256, budget=6)


def test_sixty_four_rows_two_operand_tiles():
    # R = 64 (the 3-hour configuration's rows): 448 rows, two B tiles of 224 in pass 2,
    # four row blocks in pass 1
    _case(62, P=1, Hq=14, Hkv=2, F=30, Tf=64, R_rows=64, k=100, budget=4)


def test_forty_eight_rows_three_row_blocks():
    # R = 48, G = 7: 336 rows, three row blocks in pass 1, two B tiles of 176 in pass 2
    _case(65, P=1, Hq=14, Hkv=2, F=30, Tf=50, R_rows=48, k=80, budget=4)


def test_twenty_rows_padding_inside_every_head():
    # R = 20 (padded to 32): 12 padding rows inside each head's 32, two row blocks, the
    # last warp of the second block padding only
    _case(66, P=2, Hq=28, Hkv=4, F=24, Tf=61, R_rows=20, k=90, budget=4, n_recent=2)


def test_group_of_eight_with_sixty_four_rows():
    # G = 8, R = 64: 512 rows, the largest supported
    _case(63, P=1, Hq=8, Hkv=1, F=24, Tf=50, R_rows=64, k=64, budget=3)


def test_one_row_equals_the_last_row_lists():
    ss = _ss()
    g = torch.Generator().manual_seed(64)
    keys = torch.randn(2, 2, 30 * 40, 128, generator=g).to(torch.bfloat16).cuda()
    q = torch.randn(2, 1, 8, 128, generator=g).to(torch.bfloat16).cuda()
    idx = ss.Index(2, 8, 2, 40, 30, device="cuda")
    idx.append(keys)
    a = idx.retrieve(q, k=50, budget=4, q_agg=ss.Q_MEAN_SOFTMAX)
    b = idx.retrieve(q, k=50, budget=4, q_agg=ss.Q_LAST)
    a.check()
    b.check()
    assert torch.equal(a.topk_tok, b.topk_tok)
    assert torch.allclose(a.topk_w, b.topk_w, rtol=1e-4, atol=1e-9)


def test_unsupported_shapes_are_rejected():
    ss = _ss()
    keys = torch.zeros(1, 1, 4 * 8, 128, dtype=torch.bfloat16, device="cuda")
    idx = ss.Index(1, 8, 1, 8, 4, device="cuda")
    idx.append(keys)
    q = torch.zeros(1, 65, 8, 128, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(ss.ShallowStreamError, match="UNSUPPORTED"):
        idx.retrieve(q, k=4, budget=2, q_agg=ss.Q_MEAN_SOFTMAX)
    with pytest.raises(ss.ShallowStreamError, match="UNSUPPORTED"):
        idx.retrieve(q[:, :4].contiguous(), k=4, budget=2, q_agg=ss.Q_MEAN_SOFTMAX,
                     head_agg=ss.H_MEAN)


def test_one_hour_index_sampled_lists():
    """The 1-hour workload with every question row: the oracle recomputes four sampled
    lists in full (32 rows x 705,600 keys each); all lists satisfy the invariants."""
    ss = _ss()
    from paper_2609_02780_gb300 import synth
    w = synth.PRESETS["hour1"]
    data = synth.make_workload(w, device=torch.device("cuda"))
    idx = ss.Index(w.n_layers, w.n_q_heads, w.n_kv_heads, w.tokens_per_frame, w.n_frames,
                   device="cuda")
    idx.append(data["keys"])
    res = idx.retrieve(data["q"], k=w.k, budget=w.budget, q_agg=ss.Q_MEAN_SOFTMAX)
    res.check()
    Uh, Tu = w.n_hist_units, w.tokens_per_unit
    gpu = PY.gpu_outputs(res, Uh)
    assert gpu["votes"].sum() == w.n_layers * w.n_q_heads * w.k
    assert np.allclose(gpu["list_stats"][:, 1], 1.0, atol=1e-3)
    assert abs(gpu["mass"].sum() - w.n_layers * w.n_q_heads) < 1e-2
    kb, qb = synth.bf16_bits(data["keys"]), synth.bf16_bits(data["q"])
    del data, idx
    torch.cuda.empty_cache()
    n_tok = Uh * Tu
    G = w.n_q_heads // w.n_kv_heads
    for L in (0, 33, 70, 111):
        i, h = divmod(L, w.n_q_heads)
        acc = None
        for r in range(w.n_rows):
            qe = np.zeros((w.n_layers, w.n_q_heads, 128))
            qe[i, h] = R.bf16_to_f64(qb[i, r, h])
            s = R.scores(qe, kb, n_tok, lists=[(i, h)])
            wr = R.softmax(s)
            acc = wr if acc is None else acc + wr
        alpha = acc / w.n_rows
        PY.check_topk(alpha, gpu["topk_tok"][L:L + 1], gpu["topk_w"][L:L + 1], alpha, w.k,
                      rel_tol=REL_ALPHA)
        assert abs(gpu["list_stats"][L, 0] - alpha.max()) <= REL_ALPHA * alpha.max()
    PY.check_chain(gpu, R.descriptors(kb, w.n_units, Tu), Uh, Tu, w.budget, w.pool_mult,
                   w.n_prev, w.frames_per_unit)
