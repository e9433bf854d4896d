"""Comparison of the CUDA path's outputs with the CPU oracle.

Floating point decides the per-list top-k, the pool order and the max-min picks, so
the checks are margin-aware where the two sides' rounding can legitimately differ,
and exact everywhere else:

  * top-k (Eq. 11): with theta = the oracle's n-th best score of a list and
    TOL_SCORE, the GPU's n tokens must include every token with s > theta + TOL and
    none with s < theta - TOL; its order must agree with the oracle's scores to TOL.
    TOL_SCORE = 2.5e-4 (natural-log score units) is >= 2x the fp32 error bound of a
    128-term dot product of bf16 values with |q|, |k| ~ N(0, 1) and x8 outliers.
  * weights within 2e-3 absolute of the oracle's fp64 softmax weights.
  * votes: exact, recomputed by the oracle from the GPU's own lists (chained).
  * pool: exact, recomputed by the oracle from the GPU's own votes and mass (chained).
  * max-min: each GPU pick's minimum distance within TOL_DIST of the best available
    at that step, recomputed in fp64 from the GPU's pool (chained); equal to the
    oracle's picks where no step is that close.
  * expansion / frames: exact from the GPU's picks (chained).
"""
from __future__ import annotations

import math

import numpy as np

from oracle import retrieval as R

TOL_SCORE = 2.5e-4
TOL_W = 2e-3
TOL_DIST = 1e-5
LOG2E = 1.0 / math.log(2.0)


def check_topk(s: np.ndarray, tok: np.ndarray, w_gpu: np.ndarray, w_ref: np.ndarray,
               k: int, lists=None, ids: np.ndarray | None = None, rel_tol: float = 0.0) -> dict:
    """s, w_ref: oracle scores / weights [lists][n_cand]; tok, w_gpu: GPU [lists][k].

    ids: the candidate id of each oracle column (default: the column index, i.e. token
    ids). rel_tol > 0 ranks by values whose rounding is relative (head-averaged
    weights): the band is then rel_tol * theta instead of TOL_SCORE."""
    n_tok = s.shape[1]
    n = min(k, n_tok)
    lists = range(s.shape[0]) if lists is None else lists
    pos_of = None if ids is None else {int(v): j for j, v in enumerate(ids)}
    ambiguous = 0
    for li in lists:
        row_tok = tok[li]
        assert (row_tok[n:] == -1).all(), f"list {li}: entries past n must be -1"
        if pos_of is None:
            got = row_tok[:n].astype(np.int64)
            assert (got >= 0).all() and (got < n_tok).all(), f"list {li}: token id out of range"
        else:
            assert all(int(v) in pos_of for v in row_tok[:n]), f"list {li}: unknown candidate id"
            got = np.array([pos_of[int(v)] for v in row_tok[:n]], dtype=np.int64)
        assert len(set(got.tolist())) == n, f"list {li}: duplicate tokens"
        srow = s[li]
        theta = np.partition(srow, n_tok - n)[n_tok - n]
        tol = rel_tol * abs(theta) if rel_tol > 0 else TOL_SCORE
        must = np.nonzero(srow > theta + tol)[0]
        assert np.isin(must, got).all(), f"list {li}: missed a token above the band"
        assert (srow[got] >= theta - tol).all(), f"list {li}: token below the band"
        # GPU order is (score desc, id asc) up to the score tolerance
        sg = srow[got]
        otol = rel_tol * np.abs(sg[1:]) if rel_tol > 0 else TOL_SCORE
        assert (np.diff(sg) <= otol).all(), f"list {li}: order disagrees with scores"
        wg = w_gpu[li, :n].astype(np.float64)
        assert np.abs(wg - w_ref[li, got]).max() <= TOL_W, f"list {li}: weight off"
        top = np.nonzero(srow >= theta)[0]            # the n best, ties at theta to low ids
        if len(top) > n:
            top = top[np.lexsort((top, -srow[top]))[:n]]
        ref_set = set(top.tolist())
        if ref_set != set(got.tolist()):
            ambiguous += 1
    return {"ambiguous_lists": ambiguous}


def check_stats(s: np.ndarray, list_stats: np.ndarray, lists=None) -> None:
    """GPU (M, L) in the log2 domain vs the oracle's log-sum-exp."""
    lists = range(s.shape[0]) if lists is None else lists
    for li in lists:
        srow = s[li]
        m = srow.max()
        lse = m + math.log(np.exp(srow - m).sum())
        M2, L = float(list_stats[li, 0]), float(list_stats[li, 1])
        assert abs(M2 / LOG2E - m) <= TOL_SCORE, f"list {li}: max off"
        assert abs(M2 / LOG2E + math.log(L) - lse) <= 1e-4 * max(1.0, abs(lse)), f"list {li}: lse"


def check_chain(gpu: dict, desc: np.ndarray, n_hist_units: int, tokens_per_unit: int,
                budget: int, pool_mult: int, n_prev: int, frames_per_unit: int,
                votes: np.ndarray | None = None) -> dict:
    """Votes, pool, max-min and expansion recomputed by the oracle from the GPU's own
    upstream outputs (votes: the oracle's votes from the GPU's lists, when they are not
    plain token votes)."""
    tok = gpu["topk_tok"]
    if votes is None:
        votes = R.unit_votes(tok[tok >= 0].reshape(1, -1) if (tok < 0).any() else tok,
                             n_hist_units, tokens_per_unit)
    assert np.array_equal(votes, gpu["votes"]), "votes differ"
    pool = R.vote_pool(gpu["votes"], gpu["mass"].astype(np.float64), pool_mult * budget)
    assert np.array_equal(pool, gpu["pool"]), "pool differs"
    # max-min: verify the greedy rule step by step in fp64
    D = desc[pool]
    sel = gpu["sel"]
    ranks = [int(np.nonzero(pool == u)[0][0]) for u in sel]
    assert len(sel) == min(budget, len(pool))
    close = 0
    if len(ranks):
        assert ranks[0] == 0, "max-min must start at the pool's best"
        mind = 1.0 - D @ D[0]
        taken = {0}
        for r in ranks[1:]:
            cand = [c for c in range(len(pool)) if c not in taken]
            best = max(mind[c] for c in cand)
            assert r not in taken
            assert mind[r] >= best - TOL_DIST, "max-min pick is not (near) the farthest"
            second = sorted((mind[c] for c in cand), reverse=True)
            if len(second) > 1 and second[0] - second[1] <= TOL_DIST:
                close += 1
            taken.add(r)
            mind = np.minimum(mind, 1.0 - D @ D[r])
    exp = R.expand_units(sel, n_prev)
    assert np.array_equal(exp, gpu["expanded"]), "expansion differs"
    assert np.array_equal(R.units_to_frames(exp, frames_per_unit), gpu["frames"])
    return {"close_maxmin_steps": close}


def gpu_outputs(res, n_hist_units: int) -> dict:
    c = res.counts.cpu().tolist()
    return {
        "topk_tok": res.topk_tok.cpu().numpy(),
        "topk_w": res.topk_w.cpu().numpy(),
        "list_stats": res.list_stats.cpu().numpy(),
        "votes": res.unit_votes[:n_hist_units].cpu().numpy().astype(np.int64),
        "mass": res.unit_mass[:n_hist_units].cpu().numpy(),
        "pool": res.pool[:c[0]].cpu().numpy().astype(np.int64),
        "sel": res.sel_units[:c[1]].cpu().numpy().astype(np.int64),
        "expanded": res.exp_units[:c[2]].cpu().numpy().astype(np.int64),
        "frames": res.frames_buf[:c[3]].cpu().numpy().astype(np.int64),
        "counts": c,
    }
