"""Pins of the CPU oracle (oracle/retrieval.py) against things other than itself:
a hand-worked example, closed forms, library routines, brute force and invariants.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

from oracle import retrieval as R

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "hand_example.json")


def to_bf16_bits(x) -> np.ndarray:
    """bf16 bits through torch's own rounding (a library routine, not the oracle's)."""
    t = torch.as_tensor(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


@pytest.fixture(scope="module")
def hand():
    with open(GOLDEN) as f:
        g = json.load(f)
    keys = to_bf16_bits(np.array(g["keys_layer0_head0"], np.float32))[None, None]
    q = np.stack([np.array(g["q_rows"]["row0"]), np.array(g["q_rows"]["row1"])])
    q_bits = to_bf16_bits(q.astype(np.float32))[None]          # [1][2][2][4]
    return g, keys, q_bits


# ---------------------------------------------------------------- bf16 helpers
def test_bf16_decode_known_patterns():
    bits = np.array([0x3F80, 0xC000, 0x3FC0, 0x0000, 0x8000, 0x7F80], np.uint16)
    assert list(R.bf16_to_f64(bits)) == [1.0, -2.0, 1.5, 0.0, -0.0, math.inf]


def test_bf16_rne_ties_to_even_and_matches_torch():
    one = np.float32(1.0)
    half_ulp = np.float32(2.0 ** -8)
    # 1 + 2^-8 sits halfway between 1 and 1 + 2^-7: even mantissa (1.0) wins
    assert R.bf16_to_f64(R.f32_to_bf16_rne(np.array([one + half_ulp])))[0] == 1.0
    # 1 + 3 * 2^-8 sits halfway between 1 + 2^-7 and 1 + 2^-6: 1 + 2^-6 is even
    x = np.array([one + 3 * half_ulp], np.float32)
    assert R.bf16_to_f64(R.f32_to_bf16_rne(x))[0] == 1.0 + 2.0 ** -6
    rng = np.random.default_rng(1)
    v = (rng.standard_normal(100_000) * 10.0 ** rng.integers(-5, 5, 100_000)).astype(np.float32)
    assert np.array_equal(R.f32_to_bf16_rne(v), to_bf16_bits(v))


# ---------------------------------------------------------------- hand-worked example
def test_hand_example_last_row(hand):
    g, keys, q_bits = hand
    tol = g["tolerance"]
    ex = g["last"]
    qe = R.query_effective(q_bits, R.Q_LAST)
    s = R.scores(qe, keys, 8)
    assert np.allclose(s, ex["scores"], atol=0, rtol=0)
    out = R.retrieve(keys, q_bits, n_units=4, tokens_per_unit=2, k=g["k"], budget=2,
                     pool_mult=2, n_prev=1)
    assert out["topk_tok"].tolist() == ex["topk_tok"]
    assert np.allclose(out["topk_w"], ex["topk_w"], atol=tol)
    assert out["votes"].tolist() == ex["votes"]
    assert np.allclose(out["mass"], ex["mass"], atol=tol)
    assert out["pool"].tolist() == ex["pool_mult2_budget2"]
    assert np.allclose(R.descriptors(keys, 4, 2), ex["descriptors"], atol=tol)
    assert out["sel"].tolist() == ex["sel_budget2"]
    assert out["expanded"].tolist() == ex["expanded_budget2"]
    out3 = R.retrieve(keys, q_bits, n_units=4, tokens_per_unit=2, k=g["k"], budget=3,
                      pool_mult=2, n_prev=1)
    assert out3["sel"].tolist() == ex["sel_budget3"]
    assert out3["expanded"].tolist() == ex["expanded_budget3"]
    assert out3["frames"].tolist() == ex["expanded_budget3"]


def test_hand_example_mean_logit(hand):
    g, keys, q_bits = hand
    qe = R.query_effective(q_bits, R.Q_MEAN_LOGIT)
    assert np.array_equal(qe, np.array(g["mean_logit"]["q_eff"], np.float64))
    out = R.retrieve(keys, q_bits, n_units=4, tokens_per_unit=2, k=3, budget=2,
                     pool_mult=2, q_agg=R.Q_MEAN_LOGIT)
    assert out["topk_tok"].tolist() == g["mean_logit"]["topk_tok"]


def test_hand_example_mean_heads(hand):
    g, keys, q_bits = hand
    ex = g["mean_heads"]
    out = R.retrieve(keys, q_bits, n_units=4, tokens_per_unit=2, k=3, budget=2,
                     pool_mult=2, head_agg=R.H_MEAN)
    assert np.allclose(out["alpha"][0], ex["alpha"], atol=g["tolerance"])
    assert out["topk_tok"].tolist() == ex["topk_tok"]
    assert out["votes"].tolist() == ex["votes"]
    assert np.allclose(out["mass"], ex["mass"], atol=g["tolerance"])
    assert out["pool"].tolist() == ex["pool_mult2_budget2"]


# ---------------------------------------------------------------- query rows
def test_query_modes_special_cases():
    rng = np.random.default_rng(2)
    q = to_bf16_bits(rng.standard_normal((2, 1, 4, 8)).astype(np.float32))
    assert np.array_equal(R.query_effective(q, R.Q_LAST), R.query_effective(q, R.Q_MEAN_LOGIT))
    rows = np.repeat(q, 5, axis=1)          # identical rows: the mean is that row
    assert np.array_equal(R.query_effective(rows, R.Q_MEAN_LOGIT), R.bf16_to_f64(q[:, 0]))
    distinct = to_bf16_bits(np.arange(2 * 3 * 4 * 8, dtype=np.float32).reshape(2, 3, 4, 8))
    assert np.array_equal(R.query_effective(distinct, R.Q_LAST), R.bf16_to_f64(distinct[:, 2]))


# ---------------------------------------------------------------- scores and GQA map
def test_gqa_group_mapping_and_scale():
    P, Hq, Hkv, d, N = 2, 28, 4, 128, 16
    keys = np.zeros((P, Hkv, N, d), np.float32)
    keys[1, 2, 5, 7] = 4.0          # only layer 1, key head 2, token 5, channel 7
    q = np.zeros((P, 1, Hq, d), np.float32)
    q[:, 0, :, 7] = 2.0
    s = R.scores(R.query_effective(to_bf16_bits(q)), to_bf16_bits(keys), N)
    s = s.reshape(P, Hq, N)
    hit = np.argwhere(s != 0)
    # query heads 14..20 read key head 2 (h // G with G = 7); value 2*4/sqrt(128)
    assert sorted(set(hit[:, 1].tolist())) == list(range(14, 21))
    assert set(hit[:, 0].tolist()) == {1} and set(hit[:, 2].tolist()) == {5}
    assert np.allclose(s[1, 14:21, 5], 8.0 / math.sqrt(128))


def test_scores_match_library_matmul():
    rng = np.random.default_rng(3)
    keys = to_bf16_bits(rng.standard_normal((1, 2, 50, 128)).astype(np.float32))
    q = to_bf16_bits(rng.standard_normal((1, 1, 4, 128)).astype(np.float32))
    s = R.scores(R.query_effective(q), keys, 50).reshape(4, 50)
    kt = torch.from_numpy(keys.view(np.int16)).view(torch.bfloat16).double()
    qt = torch.from_numpy(q.view(np.int16)).view(torch.bfloat16).double()
    for h in range(4):
        ref = (kt[0, h // 2] @ qt[0, 0, h]) / math.sqrt(128)
        assert np.allclose(s[h], ref.numpy(), rtol=1e-13, atol=1e-13)


# ---------------------------------------------------------------- softmax
def test_softmax_library_and_two_token_closed_form():
    import scipy.special
    rng = np.random.default_rng(4)
    s = rng.standard_normal((5, 300)) * 3
    w = R.softmax(s)
    assert np.allclose(w, scipy.special.softmax(s, axis=-1), rtol=1e-12, atol=0)
    assert np.allclose(w.sum(-1), 1.0, atol=1e-12)
    d = 1.7
    w2 = R.softmax(np.array([[d, 0.0]]))
    assert abs(w2[0, 0] - 1 / (1 + math.exp(-d))) < 1e-15
    M, L = R.log_sum_stats(s)
    assert np.allclose(M + np.log(L), scipy.special.logsumexp(s, axis=-1), rtol=1e-13)


# ---------------------------------------------------------------- top-k
def brute_topk_ok(vals, ids, sel):
    sel = list(sel)
    rest = [i for i in ids if i not in set(sel)]
    pos = {int(i): j for j, i in enumerate(ids)}
    for a in sel:
        for b in rest:
            va, vb = vals[pos[a]], vals[pos[b]]
            if not (va > vb or (va == vb and a < b)):
                return False
    for a, b in zip(sel, sel[1:]):        # emitted in (value desc, id asc) order
        va, vb = vals[pos[a]], vals[pos[b]]
        if not (va > vb or (va == vb and a < b)):
            return False
    return True


def test_topk_brute_force_small():
    rng = np.random.default_rng(5)
    for trial in range(200):
        n = int(rng.integers(1, 12))
        vals = rng.integers(-3, 4, n).astype(np.float64)   # many ties
        k = int(rng.integers(1, 14))
        sel = R.topk_rows(vals[None], k)[0]
        assert len(sel) == min(k, n)
        assert brute_topk_ok(vals, list(range(n)), sel)


def test_topk_all_equal_lowest_ids_and_k_ge_n():
    vals = np.zeros((2, 10))
    assert R.topk_rows(vals, 4).tolist() == [[0, 1, 2, 3]] * 2
    assert R.topk_rows(vals, 50)[0].tolist() == list(range(10))


# ---------------------------------------------------------------- votes and mass
def test_votes_invariants_and_k_ge_n():
    rng = np.random.default_rng(6)
    keys = to_bf16_bits(rng.standard_normal((2, 2, 40, 128)).astype(np.float32))
    q = to_bf16_bits(rng.standard_normal((2, 3, 4, 128)).astype(np.float32))
    out = R.retrieve(keys, q, n_units=10, tokens_per_unit=4, k=7, budget=2)
    assert out["votes"].sum() == 2 * 4 * 7                  # P * Hq * k
    assert np.allclose(out["mass"].sum(), 2 * 4, atol=1e-12)  # each list's weights sum to 1
    assert np.array_equal(out["votes"], np.bincount(out["topk_tok"].ravel() // 4, minlength=10))
    full = R.retrieve(keys, q, n_units=10, tokens_per_unit=4, k=1000, budget=2)
    assert full["votes"].tolist() == [2 * 4 * 4] * 10        # every token voted by every list


# ---------------------------------------------------------------- pool
def test_pool_order_ties():
    votes = np.array([3, 5, 5, 0, 3, 5])
    mass = np.array([0.1, 0.2, 0.2, 0.9, 0.3, 0.1])
    # votes 5: units 1, 2 tie on mass -> id; then 5; votes 3: 4 (0.3) then 0; then 3
    assert R.vote_pool(votes, mass, 10).tolist() == [1, 2, 5, 4, 0, 3]
    assert R.vote_pool(votes, mass, 2).tolist() == [1, 2]


# ---------------------------------------------------------------- descriptors
def test_descriptor_head_major_vec_and_norm():
    P, Hkv, d, T = 2, 3, 128, 5
    keys = np.zeros((P, Hkv, 2 * T, d), np.float32)
    keys[-1, 0, :T, 0] = 3.0
    keys[-1, 2, :T, 1] = 4.0            # unit 0: 3 at [0], 4 at [2*128 + 1]
    keys[0] = 100.0                     # other layers must not matter (final layer only)
    keys[-1, 1, T:, 5] = np.arange(T)   # unit 1: mean 2 at [128 + 5]
    D = R.descriptors(to_bf16_bits(keys), 2, T)
    e = np.zeros(Hkv * d)
    e[0], e[2 * d + 1] = 0.6, 0.8
    assert np.allclose(D[0], e, atol=1e-15)
    e1 = np.zeros(Hkv * d)
    e1[d + 5] = 1.0
    assert np.allclose(D[1], e1, atol=1e-15)
    zero = R.descriptors(to_bf16_bits(np.zeros((1, 2, 4, d), np.float32)), 2, 2)
    assert np.array_equal(zero, np.zeros((2, 2 * d)))        # Norm(0) = 0
    rng = np.random.default_rng(7)
    D2 = R.descriptors(to_bf16_bits(rng.standard_normal((2, 4, 60, 128)).astype(np.float32)), 6, 10)
    assert np.allclose(np.linalg.norm(D2, axis=1), 1.0, atol=1e-14)


# ---------------------------------------------------------------- max-min diversity
def brute_greedy_ok(pool, desc, sel):
    """Exhaustive check of the greedy max-min rule at every step."""
    D = desc[pool]
    ranks = [int(np.nonzero(pool == u)[0][0]) for u in sel]
    if ranks[0] != 0:
        return False
    for step in range(1, len(ranks)):
        chosen = ranks[:step]
        best_r, best = None, -np.inf
        for r in range(len(pool)):
            if r in chosen:
                continue
            m = min(1.0 - float(D[r] @ D[c]) for c in chosen)
            if m > best:
                best_r, best = r, m
        if best_r != ranks[step]:
            return False
    return True


def test_maxmin_brute_force_random():
    rng = np.random.default_rng(8)
    for trial in range(30):
        n = int(rng.integers(1, 15))
        desc = rng.standard_normal((n + 3, 6))
        desc /= np.linalg.norm(desc, axis=1, keepdims=True)
        pool = rng.permutation(n + 3)[:n]
        budget = int(rng.integers(1, n + 3))
        sel = R.maxmin_select(pool, desc, budget)
        assert len(sel) == min(budget, n) and len(set(sel.tolist())) == len(sel)
        assert set(sel.tolist()) <= set(pool.tolist())
        assert brute_greedy_ok(pool, desc, sel)


def test_maxmin_identical_and_orthogonal_follow_pool_order():
    pool = np.array([4, 2, 0, 3, 1])
    same = np.tile(np.array([[0.6, 0.8]]), (5, 1))
    assert R.maxmin_select(pool, same, 3).tolist() == [4, 2, 0]
    ortho = np.eye(5)
    assert R.maxmin_select(pool, ortho, 4).tolist() == [4, 2, 0, 3]


def test_maxmin_spreads_over_clusters():
    # three tight clusters of near-duplicates; the pool lists cluster A first
    rng = np.random.default_rng(9)
    centers = np.eye(3)
    desc = np.concatenate([c + 0.01 * rng.standard_normal((4, 3)) for c in centers])
    desc /= np.linalg.norm(desc, axis=1, keepdims=True)
    pool = np.arange(12)
    sel = R.maxmin_select(pool, desc, 3)
    assert sorted(u // 4 for u in sel) == [0, 1, 2]


# ---------------------------------------------------------------- expansion
def test_expand_closed_form():
    assert R.expand_units(np.array([5, 2, 0]), 1).tolist() == [0, 1, 2, 4, 5]
    assert R.expand_units(np.array([3, 4]), 1).tolist() == [2, 3, 4]
    assert R.expand_units(np.array([1, 7]), 2).tolist() == [0, 1, 5, 6, 7]
    assert R.expand_units(np.array([6]), 0).tolist() == [6]
    assert R.units_to_frames(np.array([0, 3]), 2).tolist() == [0, 1, 6, 7]


# ---------------------------------------------------------------- history split (Eq. 4)
def test_recent_units_are_never_scored_or_selected():
    rng = np.random.default_rng(10)
    keys = rng.standard_normal((1, 1, 40, 16)).astype(np.float32)
    keys[0, 0, 36:] += 50.0             # the last unit is hugely attractive ...
    q = np.ones((1, 1, 1, 16), np.float32)
    out = R.retrieve(to_bf16_bits(keys), to_bf16_bits(q), n_units=10, tokens_per_unit=4,
                     k=5, budget=3, n_recent=1)
    assert out["n_hist_units"] == 9     # ... but it is recent
    assert out["topk_tok"].max() < 36 and out["expanded"].max() < 9
    empty = R.retrieve(to_bf16_bits(keys), to_bf16_bits(q), n_units=10, tokens_per_unit=4,
                       k=5, budget=3, n_recent=10)
    assert empty["sel"].size == 0 and empty["frames"].size == 0


# ---------------------------------------------------------------- end to end sanity
def test_planted_units_are_found():
    rng = np.random.default_rng(11)
    P, Hq, Hkv, d, T, U = 2, 4, 2, 32, 8, 30
    keys = rng.standard_normal((P, Hkv, U * T, d)).astype(np.float32)
    q = rng.standard_normal((P, 2, Hq, d)).astype(np.float32)
    planted = [3, 11, 25]
    for i in range(P):
        for g in range(Hkv):
            qbar = q[i, -1, g * 2:(g + 1) * 2].mean(0)
            for u in planted:
                keys[i, g, u * T:(u + 1) * T] += 2.0 * qbar
    out = R.retrieve(to_bf16_bits(keys), to_bf16_bits(q), n_units=U, tokens_per_unit=T,
                     k=24, budget=3)
    # the planted units lead the vote-ranked pool; diversity then starts from the top
    # one (the planted units share a descriptor direction, so max-min spreads out)
    assert set(out["pool"][:3].tolist()) == set(planted)
    assert out["sel"][0] == out["pool"][0]


# ---------------------------------------------------------------- mean of the rows' softmaxes
def test_hand_example_mean_of_row_softmaxes(hand):
    g, keys, q_bits = hand
    tol = g["tolerance"]
    ex = g["mean_softmax"]
    out = R.retrieve(keys, q_bits, n_units=4, tokens_per_unit=2, k=g["k"], budget=2,
                     pool_mult=2, n_prev=1, q_agg=R.Q_MEAN_SOFTMAX)
    assert np.allclose(out["alpha"], ex["alpha"], atol=tol)
    assert out["topk_tok"].tolist() == ex["topk_tok"]
    assert out["votes"].tolist() == ex["votes"]
    assert np.allclose(out["mass"], ex["mass"], atol=tol)
    assert out["pool"].tolist() == ex["pool_mult2_budget2"]


def test_mean_of_row_softmaxes_against_library_softmax():
    sp = pytest.importorskip("scipy.special")
    rng = np.random.default_rng(11)
    P, R_, Hq, Hkv, N = 2, 3, 4, 2, 40
    keys = to_bf16_bits(rng.standard_normal((P, Hkv, N, 128)).astype(np.float32))
    q = to_bf16_bits(rng.standard_normal((P, R_, Hq, 128)).astype(np.float32))
    alpha = R.row_softmax_mean(q, keys, N)
    K = torch.tensor(R.bf16_to_f64(keys))
    Q = torch.tensor(R.bf16_to_f64(q))
    for i in range(P):
        for h in range(Hq):
            s = (Q[i, :, h] @ K[i, h // 2].T / math.sqrt(128)).numpy()   # [R][N]
            ref = sp.softmax(s, axis=1).mean(axis=0)
            assert np.allclose(alpha[i * Hq + h], ref, rtol=1e-12, atol=0)
    assert np.allclose(alpha.sum(1), 1.0, atol=1e-12)


def test_mean_of_row_softmaxes_with_one_row_is_the_last_row_softmax():
    rng = np.random.default_rng(12)
    keys = to_bf16_bits(rng.standard_normal((1, 1, 30, 128)).astype(np.float32))
    q = to_bf16_bits(rng.standard_normal((1, 1, 2, 128)).astype(np.float32))
    a = R.retrieve(keys, q, n_units=5, tokens_per_unit=6, k=7, budget=2, q_agg=R.Q_MEAN_SOFTMAX)
    b = R.retrieve(keys, q, n_units=5, tokens_per_unit=6, k=7, budget=2, q_agg=R.Q_LAST)
    assert np.allclose(a["alpha"], b["w"], rtol=1e-14)
    for key in ("topk_tok", "votes", "pool", "sel", "frames"):
        assert np.array_equal(a[key], b[key]), key
