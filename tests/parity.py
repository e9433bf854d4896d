"""Comparison of the CUDA path's outputs with the CPU oracle.

Floating point decides the per-list top-k, the pool order and the max-min picks, so
the checks are margin-aware where the two sides' rounding can legitimately differ,
and exact everywhere else:

  * top-k (Eq. 11): with theta = the oracle's n-th best score of a list and
    TOL_SCORE, the GPU's n tokens must include every token with s > theta + TOL and
    none with s < theta - TOL; its order must agree with the oracle's scores to TOL.
    TOL_SCORE = 2.5e-4 (natural-log score units) is >= 2x the fp32 error bound of a
    128-term dot product of bf16 values with |q|, |k| ~ N(0, 1) and x8 outliers.
  * weights within 2e-3 absolute and 1e-3 relative of the oracle's fp64 softmax
    weights (the absolute bound alone says little when weights are ~1e-6).
  * votes: exact, recomputed by the oracle from the GPU's own lists (chained).
  * pool: exact, recomputed by the oracle from the GPU's own votes and mass (chained).
  * max-min: each GPU pick's minimum distance within TOL_DIST of the best available
    at that step, recomputed in fp64 from the GPU's pool (chained); equal to the
    oracle's picks where no step is that close.
  * expansion / frames: exact from the GPU's picks (chained).
  * end to end: the GPU's selection and frames equal the oracle's own run from its own
    lists unless a list, a pool position or a max-min step is inside its band
    (check_end_to_end says which case held).
"""
from __future__ import annotations

import math

import numpy as np

from oracle import retrieval as R

TOL_SCORE = 2.5e-4
TOL_W = 2e-3
TOL_W_REL = 1e-3
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
        wr = w_ref[li, got]
        assert np.abs(wg - wr).max() <= TOL_W, f"list {li}: weight off"
        # and relative: a weight's error follows its score's (TOL_SCORE) and the list's
        # log-sum-exp (1e-4), so 1e-3 of the weight itself (plus a floor for underflow)
        assert (np.abs(wg - wr) <= TOL_W_REL * wr + 1e-12).all(), f"list {li}: weight off (rel)"
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


TOL_MASS = 1e-4   # relative: the GPU's unit mass against the oracle's (default path)


def _greedy_close_steps(pool: np.ndarray, desc: np.ndarray, budget: int) -> int:
    """Steps of the oracle's own max-min over `pool` whose best and second-best
    distances are within TOL_DIST (where the two sides' rounding may pick differently)."""
    n = min(budget, len(pool))
    if n <= 1:
        return 0
    D = desc[pool]
    mind = 1.0 - D @ D[0]
    taken = np.zeros(len(pool), dtype=bool)
    taken[0] = True
    close = 0
    for _ in range(n - 1):
        cand = np.nonzero(~taken)[0]
        vals = np.sort(mind[cand])[::-1]
        if len(vals) > 1 and vals[0] - vals[1] <= TOL_DIST:
            close += 1
        r = cand[np.argmax(mind[cand])]          # first maximum: the better pool rank
        taken[r] = True
        mind = np.minimum(mind, 1.0 - D @ D[r])
    return close


def _mass_near_ties(votes: np.ndarray, mass: np.ndarray, pool_n: int, rel: float) -> int:
    """Adjacent pairs in the oracle's (votes desc, mass desc, id asc) ranking, up to the
    first unit left out of the pool, with equal votes and masses within `rel`."""
    order = np.lexsort((np.arange(len(votes)), -mass, -votes))[:pool_n + 1]
    ties = 0
    for a, b in zip(order[:-1], order[1:]):
        if votes[a] == votes[b] and abs(mass[a] - mass[b]) <= rel * max(abs(mass[a]), abs(mass[b])):
            ties += 1
    return ties


def check_end_to_end(gpu: dict, ref: dict, ambiguous_lists: int, desc: np.ndarray,
                     budget: int, pool_mult: int = 4, rel_mass: float = TOL_MASS) -> str:
    """The GPU's final selection and frames against the oracle's own end-to-end run
    (ref: the oracle's votes, mass, pool, sel, frames from its own lists). They must be
    equal unless a decision on the way is inside its tolerance band: a list whose top-k
    set differs from the oracle's, a pool position decided by masses within rel_mass,
    or a max-min step decided by distances within TOL_DIST. Returns which case held."""
    votes = np.asarray(ref["votes"], np.int64)
    mass = np.asarray(ref["mass"], np.float64)
    pool_n = len(ref["pool"])
    ties = _mass_near_ties(votes, mass, pool_n, rel_mass)
    close = _greedy_close_steps(np.asarray(ref["pool"], np.int64), desc, budget)
    exact = (gpu["sel"].tolist() == list(ref["sel"]) and
             gpu["frames"].tolist() == list(ref["frames"]))
    if ambiguous_lists == 0 and ties == 0 and close == 0:
        assert exact, "end-to-end selection differs with no decision inside its band"
    if exact:
        return "e2e ids exact"
    return (f"e2e ids differ inside the bands: {ambiguous_lists} ambiguous lists, "
            f"{ties} mass near-ties, {close} close max-min steps")


def gpu_comp(cl: dict, tokens_per_frame: int, frames_per_unit: int) -> dict:
    """The GPU's compressed windows (Index.clusters()) in the oracle's form: centroid
    bits [P][Hkv][n_w][n_c][d], assignment [P][Hkv][n_w][W * T_f] gathered from each
    window's own first token, the window length and every window's first frame."""
    import torch
    WF = int(cl["window_frames"])
    Wt = WF * tokens_per_frame
    f0 = [int(u) * frames_per_unit for u in cl["window_first_unit"].cpu().tolist()]
    asg = cl["assignment"].cpu().numpy()
    A = np.stack([asg[:, :, f * tokens_per_frame:f * tokens_per_frame + Wt] for f in f0], axis=2)
    cb = cl["centroids"].detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)
    return {"centroid_bits": cb, "assign": A.astype(np.int64), "window_frames": WF,
            "window_first_frames": f0}


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
