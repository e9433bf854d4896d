"""Oracle: k-means compression of the shallow index and retrieval over centroids.

Test infrastructure only (see the package docstring).

The cluster-compressed index variant replaces, per (layer, key head), the keys of a
window of W consecutive frames by n_c centroids from Lloyd's algorithm, and
retrieval scores centroids in place of those tokens, then expands each selected
centroid to its member tokens. The paper's own compression (Sec. 4.1, Eq. 5-7:
budget-triggered online clustering of units with running-mean representative KVs,
scored by Eq. 13) is the closest text; the token-level k-means reading is:

  * X = the window's keys (exact bf16 values), C^0 = X[0:n_c] (the window's first
    tokens in token order), then `iters` rounds of
      assign  a(x) = argmin_c ||x - c||^2 (lowest centroid id on ties)
      update  c = mean of its members; a centroid with no members keeps its value.
    Members are the last round's assignment; the stored centroid is the last
    round's mean rounded to bf16.
  * Windows start on multiples of W frames but need not be adjacent: compressions
    made one after another can leave raw frames before, between and after them.
  * Retrieval candidates of a list: the centroids of every compressed window whose
    first unit is in the history, and the raw tokens of the history units that no
    compressed window covers. Softmax over all of them; top-k by (score desc, id
    asc) with centroid (w, c) given id CID_BASE + w * n_c + c, after all token ids
    (w counts windows in the order they were compressed).
  * A selected centroid gives one vote to each member token's unit (history units
    only); its weight is apportioned to units by member share |members in u| /
    |members|. Empty centroids stay candidates but vote for nothing.
"""
from __future__ import annotations

import numpy as np

from .retrieval import (bf16_to_f64, f32_to_bf16_rne, history_units, query_effective,
                        softmax, log_sum_stats, topk_rows, vote_pool, maxmin_select,
                        expand_units, units_to_frames, descriptors, H_PER_QHEAD, Q_LAST)

CID_BASE = 1 << 30


def lloyd(X: np.ndarray, n_c: int, iters: int) -> tuple[np.ndarray, np.ndarray]:
    """Lloyd's algorithm from C^0 = X[:n_c]. Returns (centroids fp64 [n_c][d],
    assignment int64 [n]) of the last round."""
    X = np.asarray(X, dtype=np.float64)
    if X.shape[0] < n_c:
        raise ValueError("window has fewer points than centroids")
    C = X[:n_c].copy()
    a = np.zeros(X.shape[0], dtype=np.int64)
    for _ in range(iters):
        a = assign(X, C)
        C = update(X, a, C)
    return C, a


def assign(X: np.ndarray, C: np.ndarray) -> np.ndarray:
    """argmin_c sum_j (x_j - c_j)^2 per point; np.argmin keeps the first (lowest id)."""
    out = np.empty(X.shape[0], dtype=np.int64)
    for s in range(0, X.shape[0], 256):
        diff = X[s:s + 256, None, :] - C[None, :, :]
        out[s:s + 256] = np.argmin((diff * diff).sum(axis=-1), axis=1)
    return out


def update(X: np.ndarray, a: np.ndarray, C_prev: np.ndarray) -> np.ndarray:
    """Mean of each centroid's members; an empty centroid keeps C_prev."""
    C = C_prev.copy()
    for c in range(C.shape[0]):
        m = a == c
        if m.any():
            C[c] = X[m].mean(axis=0)
    return C


def compress(key_bits: np.ndarray, *, tokens_per_frame: int, first_frame: int,
             n_frames: int, window_frames: int, n_centroids: int, iters: int) -> dict:
    """Compress frames [first_frame, first_frame + n_frames) in windows of
    window_frames. Returns fp64 centroids [P][Hkv][n_w][n_c][d], their bf16 bits (via
    fp32, nearest-even), and the member assignment [P][Hkv][n_w][W * T_f]."""
    if n_frames % window_frames:
        raise ValueError("n_frames must be a multiple of window_frames")
    P, Hkv, _, d = key_bits.shape
    n_w = n_frames // window_frames
    Wt = window_frames * tokens_per_frame
    C = np.empty((P, Hkv, n_w, n_centroids, d), dtype=np.float64)
    A = np.empty((P, Hkv, n_w, Wt), dtype=np.int64)
    for i in range(P):
        for g in range(Hkv):
            for w in range(n_w):
                t0 = (first_frame + w * window_frames) * tokens_per_frame
                X = bf16_to_f64(key_bits[i, g, t0:t0 + Wt])
                C[i, g, w], A[i, g, w] = lloyd(X, n_centroids, iters)
    bits = f32_to_bf16_rne(C.astype(np.float32))
    return {"centroids": C, "centroid_bits": bits, "assign": A,
            "first_frame": first_frame, "window_frames": window_frames,
            "window_first_frames": [first_frame + w * window_frames for w in range(n_w)]}


def window_first_frames(comp: dict, n_windows: int) -> list[int]:
    """First frame of every window: comp["window_first_frames"] when given (windows of
    several compressions), else adjacent windows from comp["first_frame"]."""
    if "window_first_frames" in comp:
        f = [int(x) for x in comp["window_first_frames"]]
        if len(f) != n_windows:
            raise ValueError("one first frame per window is needed")
        return f
    return [int(comp["first_frame"]) + w * int(comp["window_frames"]) for w in range(n_windows)]


def _member_units(A, i, g, w, c, win_f0, tokens_per_frame, tokens_per_unit):
    """Units of the member tokens of centroid c of window w (first frame win_f0[w]) at
    (layer i, key head g)."""
    m = np.nonzero(A[i, g, w] == c)[0]
    t = win_f0[w] * tokens_per_frame + m
    return t // tokens_per_unit


def compressed_votes(tok: np.ndarray, A: np.ndarray, *, n_q_heads: int, n_kv_heads: int,
                     n_centroids: int, window_frames: int, tokens_per_frame: int,
                     tokens_per_unit: int, n_hist_units: int, first_frame: int = 0,
                     window_first: list[int] | None = None) -> np.ndarray:
    """Unit votes of per-(layer, query head) lists that mix token ids and centroid ids:
    a token votes for its unit, a centroid once for the unit of each member token
    (history units only). A: assignments [P][Hkv][n_w][W * T_f]; window_first: the
    first frame of every window (default: adjacent windows from first_frame)."""
    G = n_q_heads // n_kv_heads
    if window_first is None:
        window_first = [first_frame + w * window_frames for w in range(A.shape[2])]
    votes = np.zeros(n_hist_units, dtype=np.int64)
    for li in range(tok.shape[0]):
        i, g = li // n_q_heads, (li % n_q_heads) // G
        for cand in tok[li]:
            cand = int(cand)
            if cand < 0:
                continue
            if cand < CID_BASE:
                votes[cand // tokens_per_unit] += 1
                continue
            w, c = divmod(cand - CID_BASE, n_centroids)
            for u in _member_units(A, i, g, w, c, window_first, tokens_per_frame,
                                   tokens_per_unit):
                if u < n_hist_units:
                    votes[u] += 1
    return votes


def retrieve_compressed(key_bits: np.ndarray, q_bits: np.ndarray, comp: dict, *,
                        n_units: int, tokens_per_unit: int, frames_per_unit: int,
                        tokens_per_frame: int, k: int, budget: int, pool_mult: int = 4,
                        n_prev: int = 1, n_recent: int = 0, q_agg: int = Q_LAST,
                        head_agg: int = H_PER_QHEAD, desc: np.ndarray | None = None,
                        centroid_bits: np.ndarray | None = None,
                        assignment: np.ndarray | None = None) -> dict:
    """Retrieval over a compressed index (see the module docstring for the reading).

    `centroid_bits` / `assignment` may be given to score another implementation's
    centroids and memberships (chained parity); they default to `comp`'s.
    """
    if head_agg != H_PER_QHEAD:
        # a centroid id names different clusters at different key heads, so a
        # head-averaged weight per centroid has no meaning
        raise ValueError("compressed retrieval is defined for per-query-head lists")
    P, Hkv, _, d = key_bits.shape
    Hq = q_bits.shape[2]
    G = Hq // Hkv
    cb = comp["centroid_bits"] if centroid_bits is None else centroid_bits
    A = comp["assign"] if assignment is None else assignment
    n_w, n_c = cb.shape[2], cb.shape[3]
    WF = comp["window_frames"]
    win_f0 = window_first_frames(comp, n_w)
    U_h = history_units(n_units, n_recent)
    if desc is None:
        desc = descriptors(key_bits, n_units, tokens_per_unit)
    qe = query_effective(q_bits, q_agg)

    # windows as unit ranges; which are candidates; which units stay detailed
    win_u0 = [f // frames_per_unit for f in win_f0]
    win_nu = WF // frames_per_unit
    covered = np.zeros(max(n_units, 1), dtype=bool)
    for u0 in win_u0:
        covered[u0:u0 + win_nu] = True
    live_w = [w for w in range(n_w) if win_u0[w] < U_h]
    raw_units = [u for u in range(U_h) if not covered[u]]
    raw_tok = np.array([u * tokens_per_unit + s for u in raw_units
                        for s in range(tokens_per_unit)], dtype=np.int64)
    cids = np.array([CID_BASE + w * n_c + c for w in live_w for c in range(n_c)],
                    dtype=np.int64)
    ids = np.concatenate([raw_tok, cids])

    n_lists = P * Hq
    s = np.empty((n_lists, len(ids)), dtype=np.float64)
    for i in range(P):
        for h in range(Hq):
            g = h // G
            kr = bf16_to_f64(key_bits[i, g, raw_tok]) if len(raw_tok) else np.zeros((0, d))
            kc = (bf16_to_f64(cb[i, g, live_w].reshape(-1, d)) if live_w
                  else np.zeros((0, d)))
            s[i * Hq + h] = np.concatenate([kr @ qe[i, h], kc @ qe[i, h]]) / np.sqrt(d)
    out = {"q_eff": qe, "n_hist_units": U_h, "ids": ids, "s": s}
    if len(ids) == 0 or U_h == 0:
        e = np.zeros(0, dtype=np.int64)
        out.update(topk_tok=np.zeros((n_lists, 0), np.int64), votes=np.zeros(U_h, np.int64),
                   mass=np.zeros(U_h), pool=e, sel=e, expanded=e, frames=e)
        return out
    w_all = softmax(s)
    M, L = log_sum_stats(s)
    pos = topk_rows(s, k, np.arange(len(ids)))            # positions into ids
    tok = ids[pos]
    tw = np.take_along_axis(w_all, pos, axis=1)

    votes = compressed_votes(tok, A, n_q_heads=Hq, n_kv_heads=Hkv, n_centroids=n_c,
                             window_frames=WF, window_first=win_f0,
                             tokens_per_frame=tokens_per_frame,
                             tokens_per_unit=tokens_per_unit, n_hist_units=U_h)
    # mass: raw weights to their unit, centroid weights by member share
    # (per window and key head: share[c][x] = members of c in the window's unit x / |c|,
    # so a list's centroid weights spread over units as w_c @ share)
    mass = np.zeros(U_h, dtype=np.float64)
    n_raw = len(raw_tok)
    raw_unit = raw_tok // tokens_per_unit
    Wt = WF * tokens_per_frame
    shares: dict[tuple[int, int, int], tuple[int, np.ndarray]] = {}

    def share_of(i, g, w):
        if (i, g, w) not in shares:
            t0 = win_f0[w] * tokens_per_frame
            u = (t0 + np.arange(Wt)) // tokens_per_unit
            u_first = int(u[0])
            cnt = np.zeros((n_c, int(u[-1]) - u_first + 1), dtype=np.float64)
            np.add.at(cnt, (A[i, g, w].astype(np.int64), u - u_first), 1.0)
            size = cnt.sum(axis=1, keepdims=True)
            shares[(i, g, w)] = (u_first, np.divide(cnt, size, out=np.zeros_like(cnt),
                                                    where=size > 0))
        return shares[(i, g, w)]

    for li in range(n_lists):
        i, g = li // Hq, (li % Hq) // G
        np.add.at(mass, raw_unit, w_all[li, :n_raw])
        for k_w, w in enumerate(live_w):
            u_first, sh = share_of(i, g, w)
            cols = slice(n_raw + k_w * n_c, n_raw + (k_w + 1) * n_c)
            add = w_all[li, cols] @ sh
            hi = min(U_h, u_first + sh.shape[1])
            mass[u_first:hi] += add[:hi - u_first]
    pool = vote_pool(votes, mass, pool_mult * budget)
    sel = maxmin_select(pool, desc, budget)
    exp = expand_units(sel, n_prev)
    out.update(M=M, L=L, w=w_all, topk_tok=tok, topk_w=tw, votes=votes, mass=mass,
               pool=pool, sel=sel, expanded=exp,
               frames=units_to_frames(exp, frames_per_unit))
    return out
