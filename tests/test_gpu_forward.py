"""Parity of the question's forward through the shallow layers (Sec. 4.2, Eq. 10) on the
GPU (through the C ABI) with the oracle.

The per-layer cases feed rows whose RMSNorm is exact on both sides (entries +-1 and +-3
in the ratio 5 : 3, so mean(h^2) = 4; norm weights 1; eps 2^-30, which vanishes next to 4
in fp32 and in the bf16 rounding of fp64): x = h / 2 exactly, so every bf16 operand the
two sides round is formed from the same inputs. Tolerances, derived from where the two
sides still round differently (the oracle is fp64):
  * q (bf16): the bf16 rounding of a value within eps = 2^-18 sum_k |x_k W_ik| (+ |b_i|,
    over the RoPE pair) of the oracle's value before rounding: the GPU's fp32
    accumulation over K = D terms errs by ~2^-24 sqrt(K) of that scale, 2^-18 leaves a
    margin, and eps stays a few percent of a bf16 step for q of order 1.
  * attention output o (Wo = identity and Wd = 0, so H_out - h_in = o exactly): the GPU
    rounds the attention weights p to bf16 (relative error <= 2^-8) for the tensor cores
    and normalises by the sum of the unrounded weights, which moves o by at most
    2^-8 sum_j p_j |v_j| <= 2^-8 (spread + |o|), spread = sum_j p_j |v_j - o| (the
    oracle's); a q or own k element at a rounding boundary moves a score by one bf16 step
    times a key entry / sqrt(d) (< 2^-8 for these inputs), the same bound again; o is
    rounded to bf16 (half a step) on the GPU: |do| <= 2^-7 (spread + |o|) + step(o) / 2.
  * MLP (Wo = 0, so H_mid = h_in and x2 = h_in / 2 exactly): H_out - h_in = a Wd^T with
    a = bf16(silu(g) u); an element of a whose oracle value lies within 1e-2 of a step of
    a rounding boundary may take the neighbouring value, so |dH_j| <= sum over those k of
    |Wd_jk| step(a_k), plus the fp32 accumulation (1e-5 of sum_k |Wd_jk| |a_k|).
  * several layers with random weights and random rows: a bf16 operand at a rounding
    boundary in layer i moves the next layer's inputs, so the check is relative (q and H
    within 2e-2 in norm); the exact parity is the per-layer cases.
"""
import numpy as np
import pytest
import torch

from oracle import forward as FW
from oracle.retrieval import bf16_to_f64
from tests.test_gpu_retrieval import run_case, to_bits

pytestmark = pytest.mark.gpu


def _ss():
    import paper_2609_02780_gb300 as ss
    return ss


def _synth():
    from paper_2609_02780_gb300 import synth
    return synth


def _np_weights(layers):
    return [{k: (None if v is None else to_bits(v)) for k, v in w.items()} for w in layers]


def _q_scale(ref, npw, n_q_heads):
    """Per element of q, sum_k |x_k| |W_ik| + |b_i| of the projection, summed over the
    RoPE pair (the rotation mixes j and j + 64)."""
    x = np.abs(ref["x"])
    W = np.abs(bf16_to_f64(npw["wqkv"]))[:n_q_heads * 128]
    sc = x @ W.T
    if npw.get("bqkv") is not None:
        sc = sc + np.abs(bf16_to_f64(npw["bqkv"]))[:n_q_heads * 128]
    sc = sc.reshape(x.shape[0], n_q_heads, 128)
    pair = sc[..., :64] + sc[..., 64:]
    return np.concatenate([pair, pair], axis=-1)


def _check_q(q_gpu_bits, q_pre, scale):
    """The GPU's q is the bf16 rounding of a value within eps = 2^-18 scale of the oracle's
    (fp32 accumulation over K = D terms, with a margin over its ~2^-24 sqrt(K) typical
    error): bf16(q_pre - eps) <= q_gpu <= bf16(q_pre + eps). Returns how many elements
    differ from the oracle's own rounding."""
    ref_bits = FW.f32_to_bf16_rne(q_pre.astype(np.float32))
    eps = 2.0 ** -18 * scale
    lo = FW.bf16_round(q_pre - eps)
    hi = FW.bf16_round(q_pre + eps)
    g = bf16_to_f64(q_gpu_bits)
    bad = (g < lo) | (g > hi)
    assert not bad.any(), (f"{int(bad.sum())} q elements outside the band, e.g. gpu "
                           f"{g[bad][:3]} oracle {q_pre[bad][:3]} eps {eps[bad][:3]}")
    return int((q_gpu_bits != ref_bits).sum())


def _bf16_step(x):
    """Spacing of bf16 values around |x| (2^(e - 7) for |x| in [2^e, 2^(e+1)))."""
    ax = np.maximum(np.abs(x), 1e-30)
    return 2.0 ** (np.floor(np.log2(ax)) - 7)


def _run(idx, layers, h_in, params):
    dev = [{k: (None if v is None else v.cuda()) for k, v in w.items()} for w in layers]
    q, h = idx.forward(dev, h_in.cuda(), params)
    torch.cuda.synchronize()
    return to_bits(q), h.cpu().double().numpy()


def _case(P, F, Tf, R, I, seed, Hkv=4, with_kv=True):
    syn = _synth()
    w = syn.PRESETS["tiny"].replace(n_layers=P, n_frames=F, tokens_per_frame=Tf, n_rows=R,
                                    n_kv_heads=Hkv, n_q_heads=Hkv * 7, seed=seed)
    q0 = syn.make_queries(w)
    keys = syn.make_keys(w, q0) if F else torch.zeros(P, Hkv, 0, 128, dtype=torch.bfloat16)
    vals = syn.make_values(w) if F else torch.zeros(P, Hkv, 0, 128, dtype=torch.bfloat16)
    layers = syn.make_forward_weights(w, I)
    h_in = syn.make_question_rows(w)
    return w, keys, vals, layers, h_in


def _exact_norm_rows(R, D, seed):
    """Rows of +-1 (5/8 of the entries) and +-3 (3/8), shuffled: mean(h^2) = 4 exactly."""
    assert D % 8 == 0
    g = torch.Generator().manual_seed(seed)
    base = torch.tensor([1.0] * (5 * D // 8) + [3.0] * (3 * D // 8))
    rows = []
    for _ in range(R):
        perm = torch.randperm(D, generator=g)
        sign = torch.randint(0, 2, (D,), generator=g) * 2.0 - 1.0
        rows.append(base[perm] * sign)
    return torch.stack(rows).to(torch.bfloat16)


EXACT_EPS = 2.0 ** -30


def _unit_norm_weights(layers):
    out = []
    for w in layers:
        w = dict(w)
        w["ln1"] = torch.ones_like(w["ln1"])
        w["ln2"] = torch.ones_like(w["ln2"])
        out.append(w)
    return out


def _near_boundary(pre, tau=1e-2):
    """Elements whose value lies within tau of a bf16 step of a rounding boundary."""
    r = FW.bf16_round(pre)
    step = _bf16_step(r)
    frac = np.abs(pre - r) / step          # 0.5 at a boundary
    return np.abs(frac - 0.5) <= tau


def _attention_layers(layers):
    """Wo = identity and Wd = 0: H_out - h_in is the attention output o (exactly)."""
    out = []
    for w in layers:
        w = dict(w)
        D = w["wo"].shape[0]
        w["wo"] = torch.eye(D, dtype=torch.bfloat16)
        w["wd"] = torch.zeros_like(w["wd"])
        out.append(w)
    return out


@pytest.mark.parametrize("R,F,Tf,kscale", [(32, 21, 64, 1), (5, 13, 50, 1), (1, 3, 64, 1),
                                            (64, 2, 200, 1), (32, 120, 196, 1),
                                            (32, 60, 196, 6)])
def test_attention_and_q_of_one_layer(R, F, Tf, kscale):
    """One layer: q (exact up to rounding boundaries) and the attention output over the
    stored tokens plus the question's own rows (bound from the bf16 attention weights).
    Covers two 128-row halves (R 32, 64), one (R 5, 1), ragged last tiles, several chunks,
    several tiles per chunk (23,520 tokens), and keys scaled by 6 so that a row's maximum
    keeps rising past the lazy margin, also between the two 64-column steps of a tile."""
    ss = _ss()
    Hkv = 4 if R != 64 else 2          # G * Rp: 224, 112, 112 (G 7), 256 (G 4 with Hq 8)
    w, keys, vals, layers, h_in = _case(1, F, Tf, R, 256, seed=R + F, Hkv=Hkv)
    if kscale != 1:
        keys = (keys.float() * kscale).to(torch.bfloat16)
    if R == 64:
        # Hq = 8, Hkv = 2 (G 4): 4 * 64 = 256 rows per key head
        syn = _synth()
        w = w.replace(n_q_heads=8)
        layers = syn.make_forward_weights(w, 256)
        h_in = syn.make_question_rows(w)
    layers = _unit_norm_weights(_attention_layers(layers))
    h_in = _exact_norm_rows(R, w.n_q_heads * 128, seed=R)
    idx = ss.Index(1, w.n_q_heads, Hkv, Tf, F, device=torch.device("cuda"))
    idx.append(keys.cuda())
    idx.append_values(vals.cuda())
    params = ss.ForwardParams(256, EXACT_EPS, 1e6)
    qb, h = _run(idx, layers, h_in, params)
    hb = to_bits(h_in)
    ref = FW.layer(bf16_to_f64(hb), _np_weights(layers)[0], to_bits(keys[0]), to_bits(vals[0]),
                   n_q_heads=w.n_q_heads, n_kv_heads=Hkv, pos0=F * Tf, eps=EXACT_EPS,
                   theta=1e6, with_spread=True)
    n_q = _check_q(qb[0], ref["q_pre"], _q_scale(ref, _np_weights(layers)[0], w.n_q_heads))
    o_gpu = h - bf16_to_f64(hb)
    tol = (2.0 ** -7 * (ref["o_spread"] + np.abs(ref["o_pre"])) * 1.01 +
           0.5 * _bf16_step(ref["o_pre"]) * 1.01 + 1e-7)
    err = np.abs(o_gpu - ref["o_pre"])
    assert (err <= tol).all(), f"attention output off by {(err / tol).max():.2f} x its bound"
    print(f"q elements at a rounding boundary: {n_q}; o error / bound max {(err / tol).max():.3f}")


@pytest.mark.parametrize("I", [384, 9856])
def test_mlp_of_one_layer_and_no_stored_tokens(I):
    """Wo = 0: H_out = h_in + bf16(silu(x2 Wg^T) (x2 Wu^T)) Wd^T; and an index with no
    stored frames (the rows attend only to each other). MLP width 384 takes the split-K
    gate/up projection and the separate SwiGLU kernel; 9856 (154 gate/up tiles of 128, one
    K split on 152 SMs) the projection with the SwiGLU product in its epilogue."""
    ss = _ss()
    w, keys, vals, layers, h_in = _case(1, 0, 64, 12, I, seed=7)
    layers = _unit_norm_weights(layers)
    for L in layers:
        L["wo"] = torch.zeros_like(L["wo"])
    h_in = _exact_norm_rows(12, 28 * 128, seed=7)
    idx = ss.Index(1, 28, 4, 64, 8, device=torch.device("cuda"))
    params = ss.ForwardParams(I, EXACT_EPS, 1e4)
    qb, h = _run(idx, layers, h_in, params)
    hb = to_bits(h_in)
    npw = _np_weights(layers)[0]
    ref = FW.layer(bf16_to_f64(hb), npw, np.zeros((4, 0, 128), np.uint16),
                   np.zeros((4, 0, 128), np.uint16), n_q_heads=28, n_kv_heads=4, pos0=0,
                   eps=EXACT_EPS, theta=1e4)
    _check_q(qb[0], ref["q_pre"], _q_scale(ref, npw, 28))
    wd = np.abs(bf16_to_f64(npw["wd"]))
    near = _near_boundary(ref["a_pre"])
    flip = (near * _bf16_step(ref["a"])) @ wd.T
    scale = np.abs(ref["a"]) @ wd.T
    tol = flip * 1.01 + 1e-5 * scale + 1e-7
    err = np.abs(h - ref["h"])
    assert (err <= tol).all(), f"MLP off by {(err / tol).max():.2f} x its bound"
    print(f"a elements at a rounding boundary: {int(near.sum())}")


def test_attention_without_stored_tokens_is_causal_over_the_rows():
    ss = _ss()
    w, keys, vals, layers, h_in = _case(1, 0, 64, 9, 256, seed=3)
    layers = _unit_norm_weights(_attention_layers(layers))
    h_in = _exact_norm_rows(9, 28 * 128, seed=3)
    idx = ss.Index(1, 28, 4, 64, 4, device=torch.device("cuda"))
    params = ss.ForwardParams(256, EXACT_EPS, 1e6, pos0=17)
    qb, h = _run(idx, layers, h_in, params)
    hb = to_bits(h_in)
    ref = FW.layer(bf16_to_f64(hb), _np_weights(layers)[0], np.zeros((4, 0, 128), np.uint16),
                   np.zeros((4, 0, 128), np.uint16), n_q_heads=28, n_kv_heads=4, pos0=17,
                   eps=EXACT_EPS, theta=1e6, with_spread=True)
    _check_q(qb[0], ref["q_pre"], _q_scale(ref, _np_weights(layers)[0], 28))
    o_gpu = h - bf16_to_f64(hb)
    # the own rows' weights stay fp32 on the GPU; q or k at a rounding boundary moves a
    # weight by < 2^-8 relative (the spread bound), then o is rounded
    tol = 2.0 ** -8 * ref["o_spread"] + 0.5 * _bf16_step(ref["o_pre"]) * 1.01 + 1e-7
    assert (np.abs(o_gpu - ref["o_pre"]) <= tol).all()


def test_three_layers_and_the_retrieval_of_their_query_rows():
    """The P-layer chain (layer offsets into the key and value slabs, per-layer weights and
    outputs), then ss_retrieve on the forward's q against the oracle's retrieval of the same
    rows."""
    ss = _ss()
    P, F, Tf, R = 3, 40, 64, 16
    w, keys, vals, layers, h_in = _case(P, F, Tf, R, 512, seed=11)
    # layer 0 takes exact-norm rows (its q is checked strictly); the rest is random
    layers[0]["ln1"] = torch.ones_like(layers[0]["ln1"])
    h_in = _exact_norm_rows(R, 28 * 128, seed=11)
    idx = ss.Index(P, 28, 4, Tf, F, device=torch.device("cuda"))
    idx.append(keys.cuda())
    idx.append_values(vals.cuda())
    params = ss.ForwardParams(512, EXACT_EPS)
    qb, h = _run(idx, layers, h_in, params)
    ref = FW.forward(to_bits(h_in), _np_weights(layers), to_bits(keys), to_bits(vals),
                     n_q_heads=28, n_kv_heads=4, eps=EXACT_EPS)
    _check_q(qb[0], ref["layers"][0]["q_pre"],
             _q_scale(ref["layers"][0], _np_weights(layers)[0], 28))
    for i in range(P):
        qg, qr = bf16_to_f64(qb[i]), bf16_to_f64(ref["q_bits"][i])
        rel = np.linalg.norm(qg - qr) / np.linalg.norm(qr)
        assert rel <= 2e-2, (i, rel)
    assert np.linalg.norm(h - ref["h"]) / np.linalg.norm(ref["h"]) <= 2e-2
    # the forward's rows are the retrieval's input
    q = torch.from_numpy(qb.view(np.int16)).view(torch.bfloat16)
    _, _, _, _, info = run_case(keys, q, tokens_per_frame=Tf, k=128, budget=6)
    print(info)


def test_wide_model_norm_in_column_chunks():
    """Hq 42 (D 5376, more columns than one CTA's threads take four at a time): the RMSNorm
    runs in column chunks with a per-row arrival count instead of one CTA per row."""
    ss = _ss()
    P, F, Tf, R, Hkv = 1, 5, 32, 4, 6
    w, keys, vals, layers, h_in = _case(P, F, Tf, R, 256, seed=17, Hkv=Hkv)
    Hq = Hkv * 7
    layers[0]["ln1"] = torch.ones_like(layers[0]["ln1"])
    h_in = _exact_norm_rows(R, Hq * 128, seed=17)
    idx = ss.Index(P, Hq, Hkv, Tf, F, device=torch.device("cuda"))
    idx.append(keys.cuda())
    idx.append_values(vals.cuda())
    params = ss.ForwardParams(256, EXACT_EPS)
    qb, h = _run(idx, layers, h_in, params)
    ref = FW.forward(to_bits(h_in), _np_weights(layers), to_bits(keys), to_bits(vals),
                     n_q_heads=Hq, n_kv_heads=Hkv, eps=EXACT_EPS)
    _check_q(qb[0], ref["layers"][0]["q_pre"],
             _q_scale(ref["layers"][0], _np_weights(layers)[0], Hq))
    assert np.linalg.norm(h - ref["h"]) / np.linalg.norm(ref["h"]) <= 2e-2


def test_bias_none_explicit_position_and_repeatability():
    ss = _ss()
    w, keys, vals, layers, h_in = _case(2, 9, 64, 7, 256, seed=5)
    for L in layers:
        L["bqkv"] = None
    idx = ss.Index(2, 28, 4, 64, 9, device=torch.device("cuda"))
    idx.append(keys.cuda())
    idx.append_values(vals.cuda())
    layers = _unit_norm_weights(layers)
    h_in = _exact_norm_rows(7, 28 * 128, seed=5)
    params = ss.ForwardParams(256, EXACT_EPS, 5e5, pos0=123_456)
    qb, h = _run(idx, layers, h_in, params)
    qb2, h2 = _run(idx, layers, h_in, params)
    assert (qb == qb2).all() and (h == h2).all()
    ref = FW.layer(bf16_to_f64(to_bits(h_in)), _np_weights(layers)[0], to_bits(keys[0]),
                   to_bits(vals[0]), n_q_heads=28, n_kv_heads=4, pos0=123_456, eps=EXACT_EPS,
                   theta=5e5)
    _check_q(qb[0], ref["q_pre"], _q_scale(ref, _np_weights(layers)[0], 28))


def test_forward_errors():
    ss = _ss()
    w, keys, vals, layers, h_in = _case(1, 4, 64, 4, 256, seed=1)
    idx = ss.Index(1, 28, 4, 64, 8, device=torch.device("cuda"))
    idx.append(keys.cuda())
    params = ss.ForwardParams(256)
    layers = [{k: (None if v is None else v.cuda()) for k, v in w.items()} for w in layers]
    with pytest.raises(ss.ShallowStreamError, match="STATE"):
        idx.forward(layers, h_in.cuda(), params)           # values missing
    idx.append_values(vals.cuda())
    with pytest.raises(ss.ShallowStreamError, match="STATE"):
        idx.append_values(vals.cuda())                     # values past the keys
    big = torch.zeros(65, 28 * 128, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(ss.ShallowStreamError, match="UNSUPPORTED"):
        idx.forward(layers, big, params)
    with pytest.raises(ss.ShallowStreamError, match="INVALID_ARG"):
        idx.forward(layers, h_in.cuda(), ss.ForwardParams(100))
    small = torch.zeros(64, dtype=torch.uint8, device="cuda")
    with pytest.raises(ss.ShallowStreamError, match="CAPACITY"):
        idx.forward(layers, h_in.cuda(), params, workspace=small)


def test_one_hour_layer_at_full_size():
    """The bench's shapes: one layer of the 1-hour stream (705,600 stored tokens per key
    head, G 7, R 32, MLP width 18944) in the launch configuration of the forward; q within
    its band and the attention output of every row and head within the bound of the bf16
    attention weights (with the per-row spread bounded by sum_j p_j |v_j| + |o|)."""
    ss = _ss()
    syn = _synth()
    w = syn.PRESETS["hour1_fwd"]
    dev = torch.device("cuda")
    keys = syn.make_keys(w, syn.make_queries(w, device=dev), device=dev)[0:1].contiguous()
    vals = syn.make_values(w, device=dev)[0:1].contiguous()
    I = w.extra["intermediate"]
    w1 = w.replace(n_layers=1)
    layers = _unit_norm_weights(_attention_layers(syn.make_forward_weights(w1, I)))
    h_in = _exact_norm_rows(w.n_rows, 28 * 128, seed=36)
    idx = ss.Index(1, 28, 4, w.tokens_per_frame, w.n_frames, device=dev)
    idx.append(keys)
    idx.append_values(vals)
    params = ss.ForwardParams(I, EXACT_EPS, 1e6)
    qb, h = _run(idx, layers, h_in, params)
    hb = to_bits(h_in)
    N = w.n_frames * w.tokens_per_frame
    npw = _np_weights(layers)[0]
    ref = FW.layer(bf16_to_f64(hb), npw, to_bits(keys[0]), to_bits(vals[0]), n_q_heads=28,
                   n_kv_heads=4, pos0=N, eps=EXACT_EPS, theta=1e6, with_spread="upper")
    n_q = _check_q(qb[0], ref["q_pre"], _q_scale(ref, npw, 28))
    o_gpu = h - bf16_to_f64(hb)
    tol = (2.0 ** -7 * (ref["o_spread"] + np.abs(ref["o_pre"])) * 1.01 +
           0.5 * _bf16_step(ref["o_pre"]) * 1.01 + 1e-7)
    err = np.abs(o_gpu - ref["o_pre"])
    assert (err <= tol).all(), f"attention output off by {(err / tol).max():.2f} x its bound"
    print(f"full size: q elements at a rounding boundary {n_q}; o error / bound max "
          f"{(err / tol).max():.3f}, median {np.median(err / tol):.4f}")
