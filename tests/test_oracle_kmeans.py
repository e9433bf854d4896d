"""Pins of the k-means compression oracle (oracle/kmeans.py): a library k-means on
separated data, the identity special case, Lloyd invariants, the reduction of
retrieval over one-token clusters to plain token retrieval, and a hand-worked
retrieval over windows that start after frame 0, leave a raw gap and hold a recent
unit (tests/golden/compressed_example.*)."""
import json
import os

import numpy as np
import pytest
import torch

from oracle import kmeans as KM
from oracle import retrieval as R


def to_bf16_bits(x) -> np.ndarray:
    t = torch.as_tensor(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def test_identity_when_every_point_is_a_centroid():
    rng = np.random.default_rng(0)
    X = rng.standard_normal((64, 128))
    C, a = KM.lloyd(X, 64, 5)
    assert a.tolist() == list(range(64))
    assert np.array_equal(C, X)


def test_matches_library_kmeans_on_separated_blobs():
    sk = pytest.importorskip("sklearn.cluster")
    rng = np.random.default_rng(1)
    centers = rng.standard_normal((8, 16)) * 20
    X = np.concatenate([c + rng.standard_normal((40, 16)) for c in centers])
    X = X[rng.permutation(len(X))]
    n_c = 8
    # start from the first n_c points, which must hit distinct blobs for a fair test
    init = X[:n_c]
    C, a = KM.lloyd(X, n_c, 5)
    km = sk.KMeans(n_clusters=n_c, init=init, n_init=1, max_iter=5, tol=0.0,
                   algorithm="lloyd").fit(X)
    counts = np.bincount(a, minlength=n_c)
    assert counts.min() > 0                      # no empty cluster: no relocation
    assert np.allclose(C, km.cluster_centers_, rtol=1e-12, atol=1e-12)


def test_lloyd_invariants():
    rng = np.random.default_rng(2)
    X = rng.standard_normal((500, 12))
    C, a = KM.lloyd(X, 16, 5)
    for c in range(16):
        m = a == c
        if m.any():
            assert np.allclose(C[c], X[m].mean(0), rtol=0, atol=1e-13)
    # inertia does not increase over Lloyd rounds
    prev = np.inf
    Cr = X[:16].copy()
    for _ in range(6):
        ar = KM.assign(X, Cr)
        inertia = ((X - Cr[ar]) ** 2).sum()
        assert inertia <= prev + 1e-9
        prev = inertia
        Cr = KM.update(X, ar, Cr)


def test_assign_ties_to_lowest_id_and_empty_keeps_centroid():
    X = np.array([[0.0, 0.0], [10.0, 0.0]])
    C = np.array([[1.0, 0.0], [-1.0, 0.0], [50.0, 50.0]])   # x0 ties c0 and c1
    a = KM.assign(X, C)
    assert a.tolist() == [0, 0]
    C2 = KM.update(X, a, C)
    assert np.allclose(C2[0], [5.0, 0.0]) and np.array_equal(C2[1:], C[1:])


def test_one_token_clusters_reduce_to_token_retrieval():
    rng = np.random.default_rng(3)
    P, Hq, Hkv, d, Tf, F = 2, 4, 2, 128, 4, 12
    keys = to_bf16_bits(rng.standard_normal((P, Hkv, F * Tf, d)).astype(np.float32))
    q = to_bf16_bits(rng.standard_normal((P, 2, Hq, d)).astype(np.float32))
    WF = 3
    comp = KM.compress(keys, tokens_per_frame=Tf, first_frame=0, n_frames=F,
                       window_frames=WF, n_centroids=WF * Tf, iters=5)
    assert np.array_equal(comp["centroid_bits"].reshape(P, Hkv, F * Tf, d), keys)
    kw = dict(n_units=F, tokens_per_unit=Tf, k=9, budget=3)
    plain = R.retrieve(keys, q, **kw)
    cmp = KM.retrieve_compressed(keys, q, comp, frames_per_unit=1, tokens_per_frame=Tf, **kw)
    # centroid (w, c) is token w * 12 + c, so ids map back and tie order is the same
    tok = np.where(cmp["topk_tok"] >= KM.CID_BASE, cmp["topk_tok"] - KM.CID_BASE,
                   cmp["topk_tok"])
    assert np.array_equal(tok, plain["topk_tok"])
    assert np.array_equal(cmp["votes"], plain["votes"])
    assert np.allclose(cmp["mass"], plain["mass"], rtol=1e-12)
    for key in ("pool", "sel", "expanded", "frames"):
        assert np.array_equal(cmp[key], plain[key]), key


def test_compressed_vote_total_is_member_count():
    rng = np.random.default_rng(4)
    P, Hq, Hkv, d, Tf, F = 1, 2, 1, 128, 8, 10
    keys = to_bf16_bits(rng.standard_normal((P, Hkv, F * Tf, d)).astype(np.float32))
    q = to_bf16_bits(rng.standard_normal((P, 1, Hq, d)).astype(np.float32))
    comp = KM.compress(keys, tokens_per_frame=Tf, first_frame=2, n_frames=6,
                       window_frames=3, n_centroids=5, iters=5)
    out = KM.retrieve_compressed(keys, q, comp, n_units=F, tokens_per_unit=Tf,
                                 frames_per_unit=1, tokens_per_frame=Tf, k=7, budget=2)
    expect = 0
    for li in range(P * Hq):
        for cand in out["topk_tok"][li]:
            if cand < KM.CID_BASE:
                expect += 1
            else:
                w, c = divmod(int(cand) - KM.CID_BASE, 5)
                expect += int((comp["assign"][0, 0, w] == c).sum())
    assert out["votes"].sum() == expect
    # candidates: 4 raw units (0, 1, 8, 9) of 8 tokens and 2 windows of 5 centroids
    assert len(out["ids"]) == 4 * 8 + 2 * 5
    assert np.allclose(out["mass"].sum(), P * Hq, atol=1e-12)   # no empty centroid here


# ---------------------------------------------------------------- hand-worked example
GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "compressed_example.json")


def _golden():
    with open(GOLDEN) as f:
        g = json.load(f)
    keys = to_bf16_bits(np.array(g["keys"], np.float32))[None, None]        # [1][1][16][4]
    q = to_bf16_bits(np.array(g["q_last_row"], np.float32))[None, None]     # [1][1][2][4]
    cb = to_bf16_bits(np.array(g["centroids"], np.float32))[None, None]     # [1][1][2][2][4]
    A = np.array(g["assignment"], np.int64)[None, None]                      # [1][1][2][4]
    comp = {"centroid_bits": cb, "assign": A, "window_frames": g["window_frames"],
            "window_first_frames": g["window_first_frames"]}
    sh = g["shape"]
    kw = dict(n_units=sh["n_units"], tokens_per_unit=sh["tokens_per_frame"] * sh["frames_per_unit"],
              frames_per_unit=sh["frames_per_unit"], tokens_per_frame=sh["tokens_per_frame"],
              k=g["k"], pool_mult=2, n_prev=1, n_recent=sh["n_recent"])
    return g, keys, q, comp, kw


def test_hand_example_compressed_retrieval():
    g, keys, q, comp, kw = _golden()
    tol = g["tolerance"]
    out = KM.retrieve_compressed(keys, q, comp, budget=2, **kw)
    assert out["ids"].tolist() == g["candidate_ids"]
    assert np.allclose(out["s"], g["scores"], atol=0, rtol=0)
    assert out["topk_tok"].tolist() == g["topk_tok"]
    assert np.allclose(out["topk_w"], g["topk_w"], atol=tol)
    assert out["votes"].tolist() == g["votes"]
    assert np.allclose(out["mass"], g["mass"], atol=tol)
    assert abs(out["mass"].sum() - g["mass_total"]) <= tol
    assert np.allclose(R.descriptors(keys, 8, 2), g["descriptors"], atol=tol)
    for key in ("pool", "sel", "expanded", "frames"):
        assert out[key].tolist() == g["budget2"][key], key
    out3 = KM.retrieve_compressed(keys, q, comp, budget=3, **kw)
    for key in ("pool", "sel", "expanded", "frames"):
        assert out3[key].tolist() == g["budget3"][key], key


def test_hand_example_compressed_votes_direct():
    g, keys, q, comp, kw = _golden()
    tok = np.array(g["topk_tok"], np.int64)
    v = KM.compressed_votes(tok, comp["assign"], n_q_heads=2, n_kv_heads=1, n_centroids=2,
                            window_frames=2, window_first=g["window_first_frames"],
                            tokens_per_frame=2, tokens_per_unit=2, n_hist_units=7)
    assert v.tolist() == g["votes"]
    # the same windows placed adjacent from frame 0 put A0's votes on units 0 and 1
    v0 = KM.compressed_votes(tok, comp["assign"], n_q_heads=2, n_kv_heads=1,
                             n_centroids=2, window_frames=2, first_frame=0,
                             tokens_per_frame=2, tokens_per_unit=2, n_hist_units=7)
    assert v0.tolist() != g["votes"]


def test_hand_example_catches_planted_mistakes(monkeypatch):
    """Plausible mistakes in the compressed path, planted in the oracle (CPU only), each
    fail the hand-worked values."""
    g, keys, q, comp, kw = _golden()

    def fails(**over) -> bool:
        out = KM.retrieve_compressed(keys, q, comp, budget=2, **kw)
        return (out["votes"].tolist() != g["votes"]
                or not np.allclose(out["mass"], g["mass"], atol=g["tolerance"]))

    assert not fails()
    # (a) the window's first frame dropped from the member-token positions
    orig = KM._member_units
    monkeypatch.setattr(KM, "_member_units",
                        lambda A, i, gg, w, c, f0, tpf, tpu: orig(A, i, gg, w, c, [0] * len(f0), tpf, tpu))
    assert fails()
    monkeypatch.setattr(KM, "_member_units", orig)
    # (b) windows taken as adjacent from the first one (the raw gap ignored)
    comp_adj = dict(comp)
    comp_adj["window_first_frames"] = [2, 4]
    out = KM.retrieve_compressed(keys, q, comp_adj, budget=2, **kw)
    assert out["votes"].tolist() != g["votes"]
    # (c) a centroid's weight spread evenly over its window's units, not by member count
    A_even = comp["assign"].copy()
    A_even[0, 0, 0] = [0, 1, 0, 1]            # A0 then has one member in each unit
    comp_even = dict(comp, assign=A_even)
    out = KM.retrieve_compressed(keys, q, comp_even, budget=2, **kw)
    assert not np.allclose(out["mass"], g["mass"], atol=g["tolerance"])
    # (d) members in the recent unit counted as votes
    tok = np.array(g["topk_tok"], np.int64)
    v8 = KM.compressed_votes(tok, comp["assign"], n_q_heads=2, n_kv_heads=1, n_centroids=2,
                             window_frames=2, window_first=g["window_first_frames"],
                             tokens_per_frame=2, tokens_per_unit=2, n_hist_units=8)
    assert v8[:7].tolist() == g["votes"] and v8[7] == 2
