"""Parity of the question's forward through the shallow layers (Sec. 4.2, Eq. 10) on the
GPU (through the C ABI) with the oracle.

Tolerances, derived from where the two sides round differently (the oracle is fp64):
  * q (bf16): equal, except an element whose oracle value before rounding lies within
    1e-2 of a bf16 step of the boundary between two bf16 values may take the other one.
    The GPU's fp32 projection differs from fp64 by ~sqrt(K) 2^-24 of its terms' scale,
    ~1e-4 of a step, so the band has a margin of ~100.
  * attention output o (layers with Wo = identity and Wd = 0, so H_out - h_in = o exactly):
    the GPU rounds the attention weights p to bf16 (relative error <= 2^-8) and normalises
    by their rounded sum, which moves o by at most 2^-8 sum_j p_j |v_j - o| (the oracle's
    "spread"); o is then rounded to bf16 (half a step) on the GPU.
  * MLP (layers with Wo = 0): H_out - h_in = bf16(silu(g) u) Wd^T; a bf16 operand that
    takes the neighbouring value (x2 near a boundary, a near a boundary) moves a term by at
    most 2^-7 of its size, and a moved x2 moves g and u by at most 2^-7 of their
    absolute-sum scale, so |dH_j| <= 2^-6 sum_k |Wd_jk| |a_k|.
  * several layers with random weights: the per-layer differences above feed the next
    layer, so the check is relative (q and H within 2e-2 in norm), the exact parity being
    the per-layer cases.
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


def _check_q(q_gpu_bits, q_pre):
    """Equal bits, or the neighbouring bf16 value with the oracle value within 1e-2 of a
    step of their midpoint."""
    ref_bits = FW.f32_to_bf16_rne(q_pre.astype(np.float32))
    diff = q_gpu_bits != ref_bits
    if diff.any():
        a = bf16_to_f64(q_gpu_bits[diff])
        b = bf16_to_f64(ref_bits[diff])
        pre = q_pre[diff]
        step = np.abs(a - b)
        # neighbours: ordered bit patterns one apart
        def ordered(bits):
            x = bits.astype(np.int64)
            return np.where(x & 0x8000, -(x & 0x7FFF), x)
        assert (np.abs(ordered(q_gpu_bits[diff]) - ordered(ref_bits[diff])) == 1).all(), \
            "q differs by more than one bf16 step"
        mid = 0.5 * (a + b)
        assert (np.abs(pre - mid) <= 1e-2 * step).all(), \
            f"q differs away from a rounding boundary: {(np.abs(pre - mid) / step).max()} steps"
    return int(diff.sum())


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


@pytest.mark.parametrize("R,F,Tf", [(32, 21, 64), (5, 13, 50), (1, 3, 64), (64, 2, 200)])
def test_attention_and_q_of_one_layer(R, F, Tf):
    """One layer: q (exact up to rounding boundaries) and the attention output over the
    stored tokens plus the question's own rows (bound from the bf16 attention weights).
    Covers two 128-row halves (R 32, 64), one (R 5, 1), ragged last tiles, several chunks."""
    ss = _ss()
    Hkv = 4 if R != 64 else 2          # G * Rp: 224, 112, 112 (G 7), 256 (G 4 with Hq 8)
    w, keys, vals, layers, h_in = _case(1, F, Tf, R, 256, seed=R + F, Hkv=Hkv)
    if R == 64:
        # Hq = 8, Hkv = 2 (G 4): 4 * 64 = 256 rows per key head
        syn = _synth()
        w = w.replace(n_q_heads=8)
        layers = syn.make_forward_weights(w, 256)
        h_in = syn.make_question_rows(w)
    layers = _attention_layers(layers)
    idx = ss.Index(1, w.n_q_heads, Hkv, Tf, F, device=torch.device("cuda"))
    idx.append(keys.cuda())
    idx.append_values(vals.cuda())
    params = ss.ForwardParams(256, 1e-6, 1e6)
    qb, h = _run(idx, layers, h_in, params)
    hb = to_bits(h_in)
    ref = FW.layer(bf16_to_f64(hb), _np_weights(layers)[0], to_bits(keys[0]), to_bits(vals[0]),
                   n_q_heads=w.n_q_heads, n_kv_heads=Hkv, pos0=F * Tf, eps=1e-6, theta=1e6,
                   with_spread=True)
    n_q = _check_q(qb[0], ref["q_pre"])
    o_gpu = h - bf16_to_f64(hb)
    tol = 2.0 ** -8 * ref["o_spread"] * 1.01 + 0.5 * _bf16_step(ref["o_pre"]) * 1.01 + 1e-7
    err = np.abs(o_gpu - ref["o_pre"])
    assert (err <= tol).all(), f"attention output off by {(err / tol).max():.2f} x its bound"
    print(f"q elements at a rounding boundary: {n_q}; o error / bound max {(err / tol).max():.3f}")


def test_mlp_of_one_layer_and_no_stored_tokens():
    """Wo = 0: H_out = h_in + bf16(silu(x2 Wg^T) (x2 Wu^T)) Wd^T; and an index with no
    stored frames (the rows attend only to each other)."""
    ss = _ss()
    w, keys, vals, layers, h_in = _case(1, 0, 64, 12, 384, seed=7)
    for L in layers:
        L["wo"] = torch.zeros_like(L["wo"])
    idx = ss.Index(1, 28, 4, 64, 8, device=torch.device("cuda"))
    params = ss.ForwardParams(384, 1e-5, 1e4)
    qb, h = _run(idx, layers, h_in, params)
    hb = to_bits(h_in)
    npw = _np_weights(layers)[0]
    ref = FW.layer(bf16_to_f64(hb), npw, np.zeros((4, 0, 128), np.uint16),
                   np.zeros((4, 0, 128), np.uint16), n_q_heads=28, n_kv_heads=4, pos0=0,
                   eps=1e-5, theta=1e4)
    _check_q(qb[0], ref["q_pre"])
    scale = np.abs(ref["a"]) @ np.abs(bf16_to_f64(npw["wd"])).T
    err = np.abs(h - ref["h"])
    assert (err <= 2.0 ** -6 * scale + 1e-6).all(), f"MLP off by {(err / (2.0 ** -6 * scale)).max()}"


def test_attention_without_stored_tokens_is_causal_over_the_rows():
    ss = _ss()
    w, keys, vals, layers, h_in = _case(1, 0, 64, 9, 256, seed=3)
    layers = _attention_layers(layers)
    idx = ss.Index(1, 28, 4, 64, 4, device=torch.device("cuda"))
    params = ss.ForwardParams(256, 1e-6, 1e6, pos0=17)
    qb, h = _run(idx, layers, h_in, params)
    hb = to_bits(h_in)
    ref = FW.layer(bf16_to_f64(hb), _np_weights(layers)[0], np.zeros((4, 0, 128), np.uint16),
                   np.zeros((4, 0, 128), np.uint16), n_q_heads=28, n_kv_heads=4, pos0=17,
                   eps=1e-6, theta=1e6, with_spread=True)
    _check_q(qb[0], ref["q_pre"])
    o_gpu = h - bf16_to_f64(hb)
    # the own rows' weights stay fp32 on the GPU: only the final rounding of o differs
    tol = 0.5 * _bf16_step(ref["o_pre"]) * 1.01 + 1e-6 * np.abs(ref["o_pre"]) + 1e-7
    assert (np.abs(o_gpu - ref["o_pre"]) <= tol).all()


def test_three_layers_and_the_retrieval_of_their_query_rows():
    """The P-layer chain (layer offsets into the key and value slabs, per-layer weights and
    outputs), then ss_retrieve on the forward's q against the oracle's retrieval of the same
    rows."""
    ss = _ss()
    P, F, Tf, R = 3, 40, 64, 16
    w, keys, vals, layers, h_in = _case(P, F, Tf, R, 512, seed=11)
    idx = ss.Index(P, 28, 4, Tf, F, device=torch.device("cuda"))
    idx.append(keys.cuda())
    idx.append_values(vals.cuda())
    params = ss.ForwardParams(512)
    qb, h = _run(idx, layers, h_in, params)
    ref = FW.forward(to_bits(h_in), _np_weights(layers), to_bits(keys), to_bits(vals),
                     n_q_heads=28, n_kv_heads=4)
    _check_q(qb[0], ref["layers"][0]["q_pre"])
    for i in range(P):
        qg, qr = bf16_to_f64(qb[i]), bf16_to_f64(ref["q_bits"][i])
        rel = np.linalg.norm(qg - qr) / np.linalg.norm(qr)
        assert rel <= 2e-2, (i, rel)
    assert np.linalg.norm(h - ref["h"]) / np.linalg.norm(ref["h"]) <= 2e-2
    # the forward's rows are the retrieval's input
    q = torch.from_numpy(qb.view(np.int16)).view(torch.bfloat16)
    _, _, _, _, info = run_case(keys, q, tokens_per_frame=Tf, k=128, budget=6)
    print(info)


def test_bias_none_explicit_position_and_repeatability():
    ss = _ss()
    w, keys, vals, layers, h_in = _case(2, 9, 64, 7, 256, seed=5)
    for L in layers:
        L["bqkv"] = None
    idx = ss.Index(2, 28, 4, 64, 9, device=torch.device("cuda"))
    idx.append(keys.cuda())
    idx.append_values(vals.cuda())
    params = ss.ForwardParams(256, 1e-6, 5e5, pos0=123_456)
    qb, h = _run(idx, layers, h_in, params)
    qb2, h2 = _run(idx, layers, h_in, params)
    assert (qb == qb2).all() and (h == h2).all()
    ref = FW.layer(bf16_to_f64(to_bits(h_in)), _np_weights(layers)[0], to_bits(keys[0]),
                   to_bits(vals[0]), n_q_heads=28, n_kv_heads=4, pos0=123_456, eps=1e-6,
                   theta=5e5)
    _check_q(qb[0], ref["q_pre"])


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
