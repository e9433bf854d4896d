"""Oracle: the paper's long-history compression of the shallow index and the cluster
evidence of a question.

Test infrastructure only (see the package docstring). Plain fp64 numpy, following
Sec. 4.1 "Optional Long-History Compression" and Sec. 4.2 (Eq. 12-13):

  * Eq. 6: units leave the detailed window oldest first. A leaving unit t with
    descriptor k_t (Eq. 3) joins the latest cluster C_j when k_t . c_j >= tau, and the
    centroid becomes c_j <- Norm((n_j c_j + k_t) / (n_j + 1)); otherwise it starts the
    next cluster with c = k_t and n = 1. The first unit to leave starts cluster 0.
  * Eq. 7: the cluster's representative keys are the running average of its members'
    keys, per layer, key head and token slot of the unit: K_j <- (n_j K_j + K_t) / (n_j + 1)
    (the index holds keys only; values are outside this path).
  * Eq. 5: the budget reading. Mem(M_T) counts the keys of the detailed units. When it
    exceeds B, the oldest detailed units beyond the near-term window (the latest
    `near_term_units` units, which include the recent ones) leave until the detailed
    keys fit B.
  * Eq. 13: each cluster's centroid is scored against the question's query state at the
    last shallow layer P - 1: score_j = (1/Hq) sum_h q_h . c_j[g(h)] / sqrt(d), with
    c_j[g] the 128 entries of key head g in the centroid (the descriptor layout). The
    top K_l clusters by (score desc, cluster id asc) are the cluster evidence.
  * Token voting, the pool, max-min and the expansion run over the detailed history
    only (Eq. 11 candidates P(S_T)): units [n_clustered, U - N_r). A selected unit's
    predecessor is added only if it is still detailed.

Parity: pinned by a hand-worked example (tests/golden/unit_clusters_example.*) and by
special cases (tau above 1: every unit its own cluster, its centroid its descriptor and
its representative its keys; tau below -1: one cluster whose representative is the plain
mean of all members' keys).
"""
from __future__ import annotations

import numpy as np

from .retrieval import (Q_LAST, Q_MEAN_LOGIT, Q_MEAN_SOFTMAX, bf16_to_f64, query_effective,
                        retrieve)


def cluster_units(desc: np.ndarray, key_bits: np.ndarray, tokens_per_unit: int,
                  units: range | list, tau: float, state: dict | None = None) -> dict:
    """Eq. 6-7 over `units` (in order) leaving the detailed window. desc [U][D] fp64
    descriptors; key_bits bf16 [P][Hkv][>= U * T_u][d]. `state` continues an earlier call
    (its last cluster may take new members). Returns the state: unit_cluster {u: j},
    centroids [C][D], counts [C], reps [C][P][Hkv][T_u][d] (fp64)."""
    Tu = tokens_per_unit
    st = {"unit_cluster": {}, "centroids": [], "counts": [], "reps": []} if state is None else {
        "unit_cluster": dict(state["unit_cluster"]),
        "centroids": [c.copy() for c in state["centroids"]],
        "counts": list(state["counts"]), "reps": [r.copy() for r in state["reps"]]}
    for t in units:
        k = np.asarray(desc[t], dtype=np.float64)
        K = bf16_to_f64(key_bits[:, :, t * Tu:(t + 1) * Tu])           # [P][Hkv][Tu][d]
        if st["centroids"] and float(k @ st["centroids"][-1]) >= tau:
            j = len(st["centroids"]) - 1
            n = st["counts"][j]
            c = (n * st["centroids"][j] + k) / (n + 1)
            nrm = np.linalg.norm(c)
            st["centroids"][j] = c / nrm if nrm > 0 else c * 0.0
            st["reps"][j] = (n * st["reps"][j] + K) / (n + 1)
            st["counts"][j] = n + 1
        else:
            j = len(st["centroids"])
            st["centroids"].append(k.copy())
            st["reps"].append(K.copy())
            st["counts"].append(1)
        st["unit_cluster"][t] = j
    return st


def units_to_leave(n_units: int, n_clustered: int, unit_key_bytes: int, budget_bytes: int,
                   near_term_units: int) -> int:
    """Eq. 5 reading: how many of the oldest detailed units leave so that the detailed
    keys fit the budget, never touching the near-term window."""
    detailed = n_units - n_clustered
    keep = max(near_term_units, budget_bytes // unit_key_bytes)
    return max(0, detailed - keep)


def cluster_scores(q_bits: np.ndarray, centroids: np.ndarray, n_kv_heads: int,
                   q_agg: int = Q_LAST) -> np.ndarray:
    """Eq. 13 scores of every cluster against the last shallow layer's query state
    (the last row, or the rows' mean for the other readings)."""
    qe = query_effective(q_bits, Q_LAST if q_agg == Q_LAST else Q_MEAN_LOGIT)[-1]   # [Hq][d]
    Hq, d = qe.shape
    G = Hq // n_kv_heads
    C = np.asarray(centroids, dtype=np.float64).reshape(len(centroids), n_kv_heads, d)
    s = np.zeros(len(centroids))
    for h in range(Hq):
        s += C[:, h // G, :] @ qe[h]
    return s / (np.sqrt(d) * Hq)


def top_clusters(scores: np.ndarray, k_l: int) -> np.ndarray:
    """The first min(k_l, C) clusters by (score desc, id asc)."""
    ids = np.arange(len(scores))
    return np.lexsort((ids, -scores))[:min(k_l, len(scores))]


def retrieve_detailed(key_bits: np.ndarray, q_bits: np.ndarray, n_clustered: int, *,
                      n_units: int, tokens_per_unit: int, frames_per_unit: int = 1,
                      k: int, budget: int, pool_mult: int = 4, n_prev: int = 1,
                      n_recent: int = 0, q_agg: int = Q_LAST, desc: np.ndarray) -> dict:
    """Token voting and diversity selection over the detailed history units
    [n_clustered, U - N_r): the plain retrieval of the detailed units, in stream numbering
    (a predecessor that has left the detailed window is not added)."""
    Tu = tokens_per_unit
    sub = key_bits[:, :, n_clustered * Tu:]
    out = retrieve(sub, q_bits, n_units=n_units - n_clustered, tokens_per_unit=Tu, k=k,
                   budget=budget, frames_per_unit=frames_per_unit, pool_mult=pool_mult,
                   n_prev=n_prev, n_recent=n_recent, q_agg=q_agg, desc=desc[n_clustered:])
    off_u = n_clustered
    res = dict(out)
    res["topk_tok"] = np.where(out["topk_tok"] >= 0, out["topk_tok"] + off_u * Tu, -1)
    for key in ("pool", "sel", "expanded"):
        res[key] = out[key] + off_u
    res["frames"] = out["frames"] + off_u * frames_per_unit
    U_h = max(0, n_units - n_recent)
    votes = np.zeros(U_h, dtype=np.int64)
    mass = np.zeros(U_h)
    votes[off_u:] = out["votes"]
    mass[off_u:] = out["mass"]
    res["votes"], res["mass"] = votes, mass
    return res
