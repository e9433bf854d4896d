"""Pins of the long-history compression oracle (oracle/unit_clusters.py): a hand-worked
example, the special cases tau > 1 (every unit its own cluster) and tau < -1 (one
cluster whose representative is the plain mean of its members), continuation across
calls, and the cluster scores against a direct restatement in torch."""
import json
import math
import os

import numpy as np
import torch

from oracle import retrieval as R
from oracle import unit_clusters as UC

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "unit_clusters_example.json")


def to_bits(x) -> np.ndarray:
    t = torch.as_tensor(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def _golden():
    with open(GOLDEN) as f:
        g = json.load(f)
    keys = to_bits(np.array(g["keys"], np.float32))[None, None]          # [1][1][16][4]
    q = to_bits(np.array(g["q_last_row"], np.float32))[None, None]       # [1][1][2][4]
    return g, keys, q


def test_hand_example_budget_clustering_and_scores():
    g, keys, q = _golden()
    tol = g["tolerance"]
    sh = g["shape"]
    desc = R.descriptors(keys, sh["n_units"], sh["tokens_per_unit"])
    n = UC.units_to_leave(sh["n_units"], 0, g["unit_key_bytes"], g["budget_bytes"],
                          g["near_term_units"])
    assert n == g["units_to_leave"]
    st = UC.cluster_units(desc, keys, sh["tokens_per_unit"], range(n), g["tau"])
    assert [st["unit_cluster"][u] for u in range(n)] == g["unit_cluster"]
    assert st["counts"] == g["counts"]
    assert np.allclose(np.array(st["centroids"]), g["centroids"], atol=tol)
    reps = np.array([r[0, 0] for r in st["reps"]])                      # [C][Tu][d]
    assert np.allclose(reps, g["reps"], atol=tol)
    sc = UC.cluster_scores(q, np.array(st["centroids"]), 1)
    assert np.allclose(sc, g["cluster_scores"], atol=tol)
    assert UC.top_clusters(sc, 2).tolist() == g["top_clusters_2"]


def test_hand_example_detailed_retrieval():
    g, keys, q = _golden()
    tol = g["tolerance"]
    sh = g["shape"]
    desc = R.descriptors(keys, sh["n_units"], sh["tokens_per_unit"])
    kw = dict(n_units=sh["n_units"], tokens_per_unit=sh["tokens_per_unit"], k=g["k"],
              pool_mult=2, n_recent=sh["n_recent"], desc=desc)
    out = UC.retrieve_detailed(keys, q, g["units_to_leave"], budget=1, **kw)
    assert out["topk_tok"].tolist() == g["topk_tok"]
    assert out["votes"].tolist() == g["votes"]
    assert np.allclose(out["mass"], g["mass"], atol=tol)
    for key in ("pool", "sel", "expanded"):
        assert out[key].tolist() == g["budget1"][key], key
    out2 = UC.retrieve_detailed(keys, q, g["units_to_leave"], budget=2, **kw)
    for key in ("sel", "expanded"):
        assert out2[key].tolist() == g["budget2"][key], key


def _random(seed, U=12, Tu=5, P=2, Hkv=2):
    rng = np.random.default_rng(seed)
    keys = to_bits(rng.standard_normal((P, Hkv, U * Tu, 128)).astype(np.float32))
    return keys, R.descriptors(keys, U, Tu), Tu


def test_tau_above_one_makes_every_unit_its_own_cluster():
    keys, desc, Tu = _random(1)
    st = UC.cluster_units(desc, keys, Tu, range(12), 1.5)
    assert [st["unit_cluster"][u] for u in range(12)] == list(range(12))
    for u in range(12):
        assert np.allclose(st["centroids"][u], desc[u])
        assert np.array_equal(st["reps"][u], R.bf16_to_f64(keys[:, :, u * Tu:(u + 1) * Tu]))


def test_tau_below_minus_one_gives_one_cluster_with_the_mean_of_its_members():
    keys, desc, Tu = _random(2)
    st = UC.cluster_units(desc, keys, Tu, range(12), -1.5)
    assert set(st["unit_cluster"].values()) == {0} and st["counts"] == [12]
    K = R.bf16_to_f64(keys).reshape(2, 2, 12, Tu, 128)
    assert np.allclose(st["reps"][0], K.mean(axis=2), rtol=0, atol=1e-12)
    # the running normalised centroid (not the normalised mean: every step renormalises)
    c = desc[0].copy()
    for n, u in enumerate(range(1, 12), start=1):
        c = (n * c + desc[u]) / (n + 1)
        c = c / np.linalg.norm(c)
    assert np.allclose(st["centroids"][0], c, atol=1e-12)


def test_continuing_across_calls_equals_one_call():
    keys, desc, Tu = _random(3)
    one = UC.cluster_units(desc, keys, Tu, range(12), 0.05)
    a = UC.cluster_units(desc, keys, Tu, range(5), 0.05)
    b = UC.cluster_units(desc, keys, Tu, range(5, 12), 0.05, state=a)
    assert b["unit_cluster"] == one["unit_cluster"] and b["counts"] == one["counts"]
    for x, y in zip(b["reps"], one["reps"]):
        assert np.allclose(x, y, atol=1e-12)


def test_cluster_scores_against_torch():
    rng = np.random.default_rng(4)
    q = to_bits(rng.standard_normal((3, 2, 8, 128)).astype(np.float32))
    cen = rng.standard_normal((9, 2 * 128))
    sc = UC.cluster_scores(q, cen, 2)
    Q = torch.tensor(R.bf16_to_f64(q[-1, -1]))                          # [8][128]
    C = torch.tensor(cen).view(9, 2, 128)
    ref = torch.stack([(C[:, h // 4] @ Q[h]) for h in range(8)]).sum(0) / (math.sqrt(128) * 8)
    assert np.allclose(sc, ref.numpy(), rtol=1e-12)
