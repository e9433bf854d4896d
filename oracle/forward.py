"""Oracle: the question's forward pass through the shallow layers (Sec. 4.2, Eq. 10).

Test infrastructure only (see the package docstring). Plain fp64 numpy.

Eq. 10 appends the question q to the retained shallow history and propagates it
through layers [0, P): layer i maps the question's hidden states H^i to H^{i+1}, its
attention reading the retained layer-i KV cache C^i_T, and yields the question's query
states Q^i_q, which the retrieval scores against the stored keys (Eq. 11). The
backbone's layers are synthetic here (no trained weights); each is a pre-norm GQA
decoder layer of the kind the evaluated backbones use:

    x   = bf16(RMSNorm(H) * w_ln1)                     RMSNorm(H) = H / sqrt(mean(H^2) + eps)
    y   = x Wqkv^T + b                                 q: Hq heads, k and v: Hkv heads of d
    q   = bf16(RoPE(y_q, pos)),  k = bf16(RoPE(y_k, pos)),  v = bf16(y_v)
    o_h = softmax_j(q_h . k_j / sqrt(d)) v_j           j over the layer's stored tokens
                                                       (keys and values as archived) and
                                                       the question's own rows up to this
                                                       one; query head h reads key head h // G
    H  += bf16(o) Wo^T
    x2  = bf16(RMSNorm(H) * w_ln2)
    H  += bf16(silu(x2 Wg^T) * (x2 Wu^T)) Wd^T

Q^i_q = q (bf16), in the [R][Hq][d] layout the retrieval takes.

Readings (listed with their reasons in the design notes):
  * RoPE: rotate-half pairs (j, j + d/2), angle = pos * theta^(-2j/d), positions
    pos0 + r for question row r; pos0 defaults to the number of stored tokens (the
    question follows the retained history). Angles are exact (fp64) on both sides.
  * rounding points: the operands of every matrix product (x, o, the MLP product, x2)
    and the outputs q, k, v are bf16 (nearest-even) on both sides; H is carried in full
    precision (fp64 here, fp32 on the GPU).
  * attention covers every stored token of the layer (history and recent units): the
    question "attends to exact full-history shallow KVs" without compression.

Parity: pinned by tests/test_oracle_forward.py: a layer without stored tokens against a
causal GQA decoder layer assembled from torch library calls (rms_norm, linear,
scaled_dot_product_attention, silu) with RoPE written as a complex rotation; stored
tokens against scaled_dot_product_attention with an explicit prefix mask; RoPE's
relative-position invariance, norm preservation and identity at position 0; zero-weight
layers.
"""
from __future__ import annotations

import numpy as np

from .retrieval import bf16_to_f64, f32_to_bf16_rne


def bf16_round(x: np.ndarray) -> np.ndarray:
    """fp64 values rounded to bf16 (nearest-even), returned as fp64. Values are first
    rounded to binary32 (nearest), which cannot change the bf16 result except for
    inputs within 2^-24 relative of a bf16 rounding boundary."""
    return bf16_to_f64(f32_to_bf16_rne(np.asarray(x, dtype=np.float64).astype(np.float32)))


def rms_norm(h: np.ndarray, w: np.ndarray, eps: float) -> np.ndarray:
    """h [R][D] -> h / sqrt(mean(h^2) + eps) * w (fp64)."""
    h = np.asarray(h, dtype=np.float64)
    inv = 1.0 / np.sqrt((h * h).mean(axis=-1, keepdims=True) + eps)
    return h * inv * np.asarray(w, dtype=np.float64)


def rope(x: np.ndarray, pos: np.ndarray, theta: float) -> np.ndarray:
    """Rotate-half RoPE. x [R][H][d] (fp64), pos [R] token positions. For j < d/2 the
    pair (x_j, x_{j+d/2}) turns by the angle pos * theta^(-2j/d)."""
    x = np.asarray(x, dtype=np.float64)
    d = x.shape[-1]
    half = d // 2
    inv = theta ** (-2.0 * np.arange(half, dtype=np.float64) / d)           # [d/2]
    ang = np.asarray(pos, dtype=np.float64)[:, None] * inv[None, :]          # [R][d/2]
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    a, b = x[..., :half], x[..., half:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def silu(x: np.ndarray) -> np.ndarray:
    x = np.asarray(x, dtype=np.float64)
    return x / (1.0 + np.exp(-x))


def attention(q: np.ndarray, hist_k: np.ndarray, hist_v: np.ndarray,
              own_k: np.ndarray, own_v: np.ndarray, spread=False):
    """q [R][Hq][d]; hist_k, hist_v [Hkv][N][d] (the layer's stored tokens); own_k, own_v
    [R][Hkv][d] (the question's rows). Row r of head h attends to the N stored tokens of
    key head h // G and to the question's rows 0..r. Returns o [R][Hq][d] (fp64); with
    spread=True also sum_j p_j |v_j - o| per element (how far a change of the weights by a
    relative e can move o: at most e times this); with spread="upper" the bound
    sum_j p_j |v_j| + |o| of it instead (one product per head, for long histories)."""
    R, Hq, d = q.shape
    Hkv = hist_k.shape[0]
    G = Hq // Hkv
    out = np.zeros((R, Hq, d), dtype=np.float64)
    spr = np.zeros((R, Hq, d), dtype=np.float64) if spread else None
    scale = 1.0 / np.sqrt(d)
    causal = np.tril(np.ones((R, R), dtype=bool))                           # row r sees 0..r
    for h in range(Hq):
        g = h // G
        keys = np.concatenate([hist_k[g], own_k[:, g]], axis=0)              # [N + R][d]
        vals = np.concatenate([hist_v[g], own_v[:, g]], axis=0)
        s = q[:, h] @ keys.T * scale                                         # [R][N + R]
        s[:, hist_k.shape[1]:][~causal] = -np.inf
        p = np.exp(s - s.max(axis=1, keepdims=True))
        p /= p.sum(axis=1, keepdims=True)
        out[:, h] = p @ vals
        if spread == "upper":
            spr[:, h] = p @ np.abs(vals) + np.abs(out[:, h])
        elif spread:
            for r in range(R):
                spr[r, h] = p[r] @ np.abs(vals - out[r, h][None, :])
    return (out, spr) if spread else out


def layer(h: np.ndarray, w: dict, hist_k_bits: np.ndarray, hist_v_bits: np.ndarray,
          *, n_q_heads: int, n_kv_heads: int, pos0: int, eps: float, theta: float,
          with_spread=False) -> dict:
    """One shallow layer F^i (Eq. 10). h [R][D] (fp64 hidden states). w: bf16 bit arrays
    ln1 [D], wqkv [(Hq + 2 Hkv) d][D], bqkv [(Hq + 2 Hkv) d] or None, wo [D][Hq d],
    ln2 [D], wgu [2 I][D] (gate rows, then up rows), wd [D][I]. hist_k_bits,
    hist_v_bits: the layer's stored keys and values, bf16 bits [Hkv][N][d].
    Returns {"h": H^{i+1} fp64, "q_bits": Q^i bf16 bits [R][Hq][d], and the intermediate
    values (q, k, v, o, a and their values before rounding)}."""
    h = np.asarray(h, dtype=np.float64)
    R, D = h.shape
    Hq, Hkv = n_q_heads, n_kv_heads
    d = D // Hq
    f = lambda name: bf16_to_f64(w[name])                                     # noqa: E731
    x = bf16_round(rms_norm(h, f("ln1"), eps))
    y = x @ f("wqkv").T
    if w.get("bqkv") is not None:
        y = y + f("bqkv")
    pos = pos0 + np.arange(R)
    yq = y[:, :Hq * d].reshape(R, Hq, d)
    yk = y[:, Hq * d:(Hq + Hkv) * d].reshape(R, Hkv, d)
    yv = y[:, (Hq + Hkv) * d:].reshape(R, Hkv, d)
    q_pre = rope(yq, pos, theta)
    q = bf16_round(q_pre)
    k = bf16_round(rope(yk, pos, theta))
    v = bf16_round(yv)
    att = attention(q, bf16_to_f64(hist_k_bits), bf16_to_f64(hist_v_bits), k, v,
                    spread=with_spread)
    o_pre, o_spread = att if with_spread else (att, None)
    o = bf16_round(o_pre.reshape(R, Hq * d))
    h1 = h + o @ f("wo").T
    x2 = bf16_round(rms_norm(h1, f("ln2"), eps))
    wgu = f("wgu")
    I = wgu.shape[0] // 2
    g = x2 @ wgu[:I].T
    u = x2 @ wgu[I:].T
    a = bf16_round(silu(g) * u)
    h2 = h1 + a @ f("wd").T
    return {"h": h2, "h_mid": h1, "q_bits": f32_to_bf16_rne(q.astype(np.float32)),
            "q": q, "q_pre": q_pre, "k": k, "v": v, "o": o, "o_pre": o_pre.reshape(R, Hq * d),
            "o_spread": None if o_spread is None else o_spread.reshape(R, Hq * d),
            "x": x, "x2": x2, "a": a, "a_pre": silu(g) * u}


def forward(h_in_bits: np.ndarray, layers: list, key_bits: np.ndarray, value_bits: np.ndarray,
            *, n_q_heads: int, n_kv_heads: int, pos0: int | None = None,
            eps: float = 1e-6, theta: float = 1e6) -> dict:
    """Eq. 10 over layers [0, P): h_in_bits bf16 bits [R][D] (the question's embedded
    rows); layers: P weight dicts (see layer); key_bits, value_bits: the index's stored
    keys and values, bf16 bits [P][Hkv][N][d]. pos0 defaults to N.
    Returns {"q_bits": [P][R][Hq][d], "h": H^P [R][D] fp64, "layers": per-layer dicts}."""
    N = key_bits.shape[2]
    p0 = N if pos0 is None else pos0
    h = bf16_to_f64(h_in_bits)
    outs = []
    for i, w in enumerate(layers):
        r = layer(h, w, key_bits[i], value_bits[i], n_q_heads=n_q_heads,
                  n_kv_heads=n_kv_heads, pos0=p0, eps=eps, theta=theta)
        outs.append(r)
        h = r["h"]
    return {"q_bits": np.stack([r["q_bits"] for r in outs]), "h": h, "layers": outs}
