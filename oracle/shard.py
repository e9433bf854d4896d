"""Oracle: one shard's share of a retrieval over an index split by token range.

Test infrastructure only (see the package docstring).

A stream's history units are split into contiguous ranges, one per GPU. For its range
[unit_begin, unit_begin + n_units) a shard scores its own keys (Sec. 4.2 scored Q-K
attention) and reports what the rest of the retrieval needs from it:

  * per list, its own top-k tokens (score desc, stream token id asc) with their scores:
    every token of a list's global top-k is in the top-k of the shard holding it;
  * per list, (M, L) over its tokens: M = max s2, L = sum 2^(s2 - M);
  * per (list, unit), (m_u, l_u) over the unit's tokens, from which the attention mass
    of a unit (its weights summed over all its tokens and all lists) follows once the
    lists' global (M, L) are known;
  * the unit descriptors of its units (Eq. 3), for the max-min step.

Scores are reported in the library's log2 domain, s2 = s * log2(e) with s = q.k / sqrt(d),
so that softmax weights are 2^(s2 - M) / L. Everything here is fp64 from the same
definitions as retrieval.py.

Parity: pinned by the merge of shard payloads reproducing the unsharded retrieval of
retrieval.py (tests/test_shard_merge.py), on two and four shards of uneven sizes.
"""
from __future__ import annotations

import numpy as np

from .retrieval import Q_LAST, descriptors, query_effective, scores

LOG2E = 1.0 / np.log(2.0)


def shard_payload(key_bits: np.ndarray, q_bits: np.ndarray, *, unit_begin: int,
                  n_units: int, tokens_per_unit: int, k: int, q_agg: int = Q_LAST) -> dict:
    """key_bits: bf16 bits [P][Hkv][>= n_units * T_u][d], the shard's own keys (its unit 0
    is stream unit unit_begin); q_bits: the question's rows [P][R][Hq][d]."""
    Tu = tokens_per_unit
    n_tok = n_units * Tu
    qe = query_effective(q_bits, q_agg)
    P, Hq = qe.shape[0], qe.shape[1]
    n_lists = P * Hq
    s2 = scores(qe, key_bits, n_tok) * LOG2E                  # [lists][n_tok]
    tok0 = unit_begin * Tu
    kk = min(k, n_tok)
    top_tok = np.full((n_lists, k), -1, dtype=np.int64)
    top_s = np.full((n_lists, k), -np.inf)
    ids = np.arange(n_tok)
    for li in range(n_lists):
        order = np.lexsort((ids, -s2[li]))[:kk]
        top_tok[li, :kk] = order + tok0
        top_s[li, :kk] = s2[li, order]
    M = s2.max(axis=1) if n_tok else np.full(n_lists, -np.inf)
    L = np.exp2(s2 - M[:, None]).sum(axis=1) if n_tok else np.zeros(n_lists)
    per_unit = s2.reshape(n_lists, n_units, Tu)
    m_u = per_unit.max(axis=2)
    l_u = np.exp2(per_unit - m_u[:, :, None]).sum(axis=2)
    return {"unit_begin": unit_begin, "n_units": n_units, "topk_tok": top_tok,
            "topk_s": top_s, "list_stats": np.stack([M, L], axis=1),
            "unit_stats": np.stack([m_u, l_u], axis=2),
            "desc": descriptors(key_bits, n_units, Tu)}
