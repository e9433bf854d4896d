"""Oracle: query-time evidence retrieval over the shallow key index (fp64 numpy).

Test infrastructure only (see the package docstring). Parity status of each function
is stated in its docstring; every function here is pinned by tests/test_oracle_*.py.

Notation (Sec. 3-4): P shallow layers, Hq query heads, Hkv key heads, G = Hq / Hkv
(query head h reads key head h // G), d head dim, T_u tokens per unit, U stored units,
N_r recent units. Token id p = unit * T_u + slot within the unit.

Readings of points the paper leaves open (each is listed with its reason in the
design notes):
  * query representation: the last question row ("final prompt token", Sec. 4.2 and
    Table 4) by default; optionally the row mean, whose logit is the mean logit.
    The row mean is formed in fp32 in row order and rounded to bf16 (nearest-even),
    a defined step that both sides take. Third option: every question row attends on
    its own and a list's weight of a token is the mean over the rows of the rows'
    softmax weights (row_softmax_mean); the list ranks tokens by that mean weight.
  * scale 1/sqrt(d) on post-RoPE q and k; softmax over the candidate history tokens.
  * per-query-head lists (P * Hq lists of k tokens) by default; "average over heads"
    (Eq. 11 as printed) as the mean of the per-head softmax weights, P lists.
  * ties: (score desc, token id asc) everywhere.
  * attention mass of a unit: the sum of its tokens' normalised weights over all
    lists (all tokens, not just the voted ones); it breaks vote ties, then unit id.
  * pool = min(pool_mult * K, |history|) units; max-min starts from the top
    vote-ranked unit, distance 1 - cosine, ties to the better pool rank.
  * expansion adds the n_prev preceding units of each selected unit (Table 4: 1).
  * Norm(0) = 0: a unit whose mean key is zero gets the zero descriptor (distance 1
    to every unit), since Eq. 3's normalisation is undefined there.
"""
from __future__ import annotations

import numpy as np

Q_LAST, Q_MEAN_LOGIT, Q_MEAN_SOFTMAX = 0, 1, 2
H_PER_QHEAD, H_MEAN = 0, 1


# ---------------------------------------------------------------------------
# bf16 <-> float (bf16 is the upper half of an IEEE-754 binary32)
# ---------------------------------------------------------------------------
def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact value of bf16 bit patterns, as float64."""
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return b.view(np.float32).astype(np.float64)


def f32_to_bf16_rne(x: np.ndarray) -> np.ndarray:
    """Round binary32 values to bf16 bit patterns, nearest-even (NaN stays NaN)."""
    x = np.asarray(x, dtype=np.float32)
    b = x.view(np.uint32).astype(np.uint64)
    lsb = (b >> np.uint64(16)) & np.uint64(1)
    r = ((b + np.uint64(0x7FFF) + lsb) >> np.uint64(16)).astype(np.uint16)
    nan = np.isnan(x)
    if nan.any():
        r = np.where(nan, ((b >> np.uint64(16)) | np.uint64(0x40)).astype(np.uint16), r)
    return r


# ---------------------------------------------------------------------------
# Query representation (Sec. 4.2 "final prompt token"; Table 4 "last prompt token")
# ---------------------------------------------------------------------------
def query_effective(q_bits: np.ndarray, mode: int = Q_LAST) -> np.ndarray:
    """q_eff[P][Hq][d] (float64) from question rows q[P][R][Hq][d] (bf16 bits).

    Q_LAST: the last row. Q_MEAN_LOGIT: the rows' mean; since a logit is linear in q,
    its logit is the mean of the rows' logits. The mean is summed in fp32 in row
    order, divided by R in fp32 and rounded to bf16 (nearest-even).
    """
    q_bits = np.asarray(q_bits, dtype=np.uint16)
    R = q_bits.shape[1]
    if R < 1:
        raise ValueError("need at least one question row")
    if mode == Q_LAST:
        return bf16_to_f64(q_bits[:, R - 1])
    if mode == Q_MEAN_LOGIT:
        x = bf16_to_f64(q_bits).astype(np.float32)
        acc = np.zeros(x[:, 0].shape, dtype=np.float32)
        for r in range(R):
            acc = (acc + x[:, r]).astype(np.float32)
        mean = (acc / np.float32(R)).astype(np.float32)
        return bf16_to_f64(f32_to_bf16_rne(mean))
    raise ValueError(f"unknown query mode {mode}")


# ---------------------------------------------------------------------------
# History (Eq. 4): the latest N_r units are recent; the rest is history
# ---------------------------------------------------------------------------
def history_units(n_units: int, n_recent: int) -> int:
    """Number of history units |H_T| = U - N_r (never negative); history = [0, U-N_r)."""
    return max(0, n_units - n_recent)


# ---------------------------------------------------------------------------
# Scored Q-K attention (Sec. 4.2) over the history tokens
# ---------------------------------------------------------------------------
def scores(q_eff: np.ndarray, key_bits: np.ndarray, n_hist_tokens: int,
           lists: list[tuple[int, int]] | None = None) -> np.ndarray:
    """s[list][p] = q_eff[i][h] . K[i][h // G][p] / sqrt(d) for p < n_hist_tokens.

    q_eff: float64 [P][Hq][d]; key_bits: bf16 bits [P][Hkv][N][d]. Lists default to all
    (i, h) in layer-major order (list id i * Hq + h). The dot product is an fp64
    matrix product of the exact bf16 values.
    """
    P, Hq, d = q_eff.shape
    Hkv = key_bits.shape[1]
    G = Hq // Hkv
    if lists is None:
        lists = [(i, h) for i in range(P) for h in range(Hq)]
    out = np.empty((len(lists), n_hist_tokens), dtype=np.float64)
    cache: dict[tuple[int, int], np.ndarray] = {}
    for li, (i, h) in enumerate(lists):
        g = h // G
        if (i, g) not in cache:
            cache.clear()
            cache[(i, g)] = bf16_to_f64(key_bits[i, g, :n_hist_tokens])
        out[li] = cache[(i, g)] @ q_eff[i, h] / np.sqrt(d)
    return out


def row_softmax_mean(q_bits: np.ndarray, key_bits: np.ndarray, n_hist_tokens: int) -> np.ndarray:
    """alpha[list][p] = (1/R) sum_r softmax_p(q_r . k_p / sqrt(d)) per (layer, query head)
    list: the mean over the question rows of each row's attention weights (Sec. 4.2's
    scored Q-K attention, taken for every question row instead of the last one).
    q_bits: bf16 bits [P][R][Hq][d]."""
    q_bits = np.asarray(q_bits, dtype=np.uint16)
    R = q_bits.shape[1]
    acc = None
    for r in range(R):
        w = softmax(scores(bf16_to_f64(q_bits[:, r]), key_bits, n_hist_tokens))
        acc = w if acc is None else acc + w
    return acc / R


def softmax(s: np.ndarray) -> np.ndarray:
    """Row softmax in fp64: exp(s - max) / sum."""
    if s.shape[-1] == 0:
        return s.copy()
    m = s.max(axis=-1, keepdims=True)
    e = np.exp(s - m)
    return e / e.sum(axis=-1, keepdims=True)


def log_sum_stats(s: np.ndarray) -> tuple[np.ndarray, np.ndarray]:
    """Per row: M = max s and L = sum exp(s - M) (natural-log domain)."""
    m = s.max(axis=-1)
    return m, np.exp(s - m[:, None]).sum(axis=-1)


# ---------------------------------------------------------------------------
# Top-M per list (Eq. 11), ties to the lower token id
# ---------------------------------------------------------------------------
def topk_rows(vals: np.ndarray, k: int, ids: np.ndarray | None = None) -> np.ndarray:
    """Per row: the first min(k, n) ids sorted by (value desc, id asc)."""
    n = vals.shape[-1]
    if ids is None:
        ids = np.arange(n)
    kk = min(k, n)
    out = np.empty((vals.shape[0], kk), dtype=np.int64)
    for r in range(vals.shape[0]):
        order = np.lexsort((ids, -vals[r]))
        out[r] = ids[order[:kk]]
    return out


# ---------------------------------------------------------------------------
# Unit votes and attention mass (Sec. 4.2, below Eq. 11)
# ---------------------------------------------------------------------------
def unit_votes(topk_tok: np.ndarray, n_hist_units: int, tokens_per_unit: int) -> np.ndarray:
    """v_t = number of (list, selected token) pairs whose token lies in unit t."""
    v = np.zeros(n_hist_units, dtype=np.int64)
    for row in np.asarray(topk_tok):
        for p in row:
            v[int(p) // tokens_per_unit] += 1
    return v


def unit_mass(weights: np.ndarray, n_hist_units: int, tokens_per_unit: int) -> np.ndarray:
    """Sum of each unit's token weights over every list and every token of the unit."""
    w = np.asarray(weights, dtype=np.float64)
    return w.reshape(w.shape[0], n_hist_units, tokens_per_unit).sum(axis=(0, 2))


# ---------------------------------------------------------------------------
# Vote-ranked pool (Sec. 4.2: top 4K by votes, ties by attention mass)
# ---------------------------------------------------------------------------
def vote_pool(votes: np.ndarray, mass: np.ndarray, pool_n: int) -> np.ndarray:
    """First min(pool_n, U_h) units by (votes desc, mass desc, unit id asc)."""
    U = len(votes)
    order = np.lexsort((np.arange(U), -np.asarray(mass, np.float64),
                        -np.asarray(votes, np.int64)))
    return order[:min(pool_n, U)].astype(np.int64)


# ---------------------------------------------------------------------------
# Unit descriptor (Eq. 3)
# ---------------------------------------------------------------------------
def descriptors(key_bits: np.ndarray, n_units: int, tokens_per_unit: int) -> np.ndarray:
    """k_t = Norm(mean over the unit's tokens of vec over key heads of K^{P-1}).

    key_bits: bf16 bits [P][Hkv][N][d]. Returns float64 [n_units][Hkv * d]; the vec
    order is key head major (head 0's d values, then head 1's, ...).
    """
    last = bf16_to_f64(key_bits[-1])                      # [Hkv][N][d]
    Hkv, N, d = last.shape
    out = np.empty((n_units, Hkv * d), dtype=np.float64)
    for u in range(n_units):
        sl = last[:, u * tokens_per_unit:(u + 1) * tokens_per_unit, :]
        mean = sl.mean(axis=1).reshape(Hkv * d)
        nrm = np.linalg.norm(mean)
        out[u] = mean / nrm if nrm > 0 else 0.0     # a zero mean has no direction
    return out


# ---------------------------------------------------------------------------
# Max-min diversity (DivTopK, Sec. 4.2 and Eq. 12)
# ---------------------------------------------------------------------------
def maxmin_select(pool: np.ndarray, desc: np.ndarray, budget: int) -> np.ndarray:
    """Greedy max-min over the pool in descriptor space.

    Start with the top vote-ranked unit; then repeatedly add the unselected pool unit
    whose minimum distance 1 - k_c . k_s to the selected set is largest (ties to the
    better pool rank), until min(budget, |pool|) units are chosen. Returns units in
    selection order.
    """
    pool = np.asarray(pool, dtype=np.int64)
    n = min(budget, len(pool))
    if n == 0:
        return np.zeros(0, dtype=np.int64)
    D = desc[pool]
    chosen = [0]
    mind = 1.0 - D @ D[0]
    taken = np.zeros(len(pool), dtype=bool)
    taken[0] = True
    while len(chosen) < n:
        best, best_r = -np.inf, -1
        for r in range(len(pool)):
            if not taken[r] and mind[r] > best:
                best, best_r = mind[r], r
        chosen.append(best_r)
        taken[best_r] = True
        mind = np.minimum(mind, 1.0 - D @ D[best_r])
    return pool[chosen]


# ---------------------------------------------------------------------------
# Temporal expansion and ordering (Eq. 12; dedup + temporal order after Eq. 13)
# ---------------------------------------------------------------------------
def expand_units(selected: np.ndarray, n_prev: int) -> np.ndarray:
    """Selected units plus their n_prev preceding units (>= 0), deduplicated, ascending."""
    s = set()
    for u in np.asarray(selected, dtype=np.int64):
        u = int(u)
        s.add(u)
        for j in range(1, n_prev + 1):
            if u - j >= 0:
                s.add(u - j)
    return np.array(sorted(s), dtype=np.int64)


def units_to_frames(units: np.ndarray, frames_per_unit: int) -> np.ndarray:
    return np.array([u * frames_per_unit + f for u in units
                     for f in range(frames_per_unit)], dtype=np.int64)


# ---------------------------------------------------------------------------
# Downstream of the per-list selections: votes -> pool -> max-min -> expansion
# ---------------------------------------------------------------------------
def select_from_lists(topk_tok: np.ndarray, mass: np.ndarray, desc: np.ndarray,
                      n_hist_units: int, tokens_per_unit: int, budget: int,
                      pool_mult: int, n_prev: int, frames_per_unit: int) -> dict:
    """Steps after Eq. 11 given per-list selections and per-unit attention mass."""
    votes = unit_votes(topk_tok, n_hist_units, tokens_per_unit)
    pool = vote_pool(votes, mass, pool_mult * budget)
    sel = maxmin_select(pool, desc, budget)
    exp = expand_units(sel, n_prev)
    return {"votes": votes, "mass": np.asarray(mass, np.float64), "pool": pool,
            "sel": sel, "expanded": exp, "frames": units_to_frames(exp, frames_per_unit)}


def retrieve(key_bits: np.ndarray, q_bits: np.ndarray, *, n_units: int,
             tokens_per_unit: int, k: int, budget: int, frames_per_unit: int = 1,
             pool_mult: int = 4, n_prev: int = 1, n_recent: int = 0,
             q_agg: int = Q_LAST, head_agg: int = H_PER_QHEAD,
             desc: np.ndarray | None = None) -> dict:
    """End-to-end query-time evidence retrieval (Sec. 4.2, Eq. 11-12).

    key_bits bf16 [P][Hkv][>= n_units*T_u][d]; q_bits bf16 [P][R][Hq][d].
    Returns the per-list selections (token ids and normalised weights, sorted by
    score desc / id asc), the softmax stats, votes, mass, pool, selection, expanded
    units and frames.
    """
    P, Hkv = key_bits.shape[0], key_bits.shape[1]
    Hq = q_bits.shape[2]
    if Hq % Hkv:
        raise ValueError("Hq must be a multiple of Hkv")
    U_h = history_units(n_units, n_recent)
    n_tok = U_h * tokens_per_unit
    if desc is None:
        desc = descriptors(key_bits, n_units, tokens_per_unit)
    if q_agg == Q_MEAN_SOFTMAX:
        if head_agg != H_PER_QHEAD:
            raise ValueError("the mean of the rows' softmaxes is defined for per-query-head lists")
        out = {"n_hist_units": U_h}
        if U_h == 0:
            empty = np.zeros(0, dtype=np.int64)
            out.update(topk_tok=np.zeros((P * Hq, 0), np.int64), topk_w=np.zeros((0, 0)),
                       votes=empty, mass=np.zeros(0), pool=empty, sel=empty, expanded=empty,
                       frames=empty)
            return out
        alpha = row_softmax_mean(q_bits, key_bits, n_tok)          # [P*Hq][n_tok]
        tok = topk_rows(alpha, k)
        out.update(alpha=alpha, topk_tok=tok, topk_w=np.take_along_axis(alpha, tok, axis=1))
        out.update(select_from_lists(tok, unit_mass(alpha, U_h, tokens_per_unit), desc, U_h,
                                     tokens_per_unit, budget, pool_mult, n_prev,
                                     frames_per_unit))
        return out
    qe = query_effective(q_bits, q_agg)
    out = {"q_eff": qe, "n_hist_units": U_h}
    if U_h == 0:
        empty = np.zeros(0, dtype=np.int64)
        out.update(topk_tok=np.zeros((P * Hq if head_agg == H_PER_QHEAD else P, 0),
                                     np.int64),
                   topk_w=np.zeros((0, 0)), votes=empty, mass=np.zeros(0), pool=empty,
                   sel=empty, expanded=empty, frames=empty)
        return out
    s = scores(qe, key_bits, n_tok)                        # [P*Hq][n_tok]
    w = softmax(s)
    M, L = log_sum_stats(s)
    out.update(s=s, w=w, M=M, L=L)
    if head_agg == H_PER_QHEAD:
        lists_val = s
        weights = w
    elif head_agg == H_MEAN:
        alpha = w.reshape(P, Hq, n_tok).mean(axis=1)        # [P][n_tok]
        lists_val = alpha
        weights = alpha
        out["alpha"] = alpha
    else:
        raise ValueError(f"unknown head aggregation {head_agg}")
    tok = topk_rows(lists_val, k)
    tw = np.take_along_axis(weights, tok, axis=1)
    mass = unit_mass(weights, U_h, tokens_per_unit)
    out.update(topk_tok=tok, topk_w=tw)
    out.update(select_from_lists(tok, mass, desc, U_h, tokens_per_unit, budget,
                                 pool_mult, n_prev, frames_per_unit))
    return out
