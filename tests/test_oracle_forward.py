"""Pins of the oracle's question forward (Sec. 4.2, Eq. 10): library routines, a second
formulation of RoPE, invariants and special cases.

The reference decoder below is assembled from torch library calls (rms_norm, linear,
scaled_dot_product_attention with GQA, silu); RoPE is written as a rotation of complex
numbers, a different formulation from the oracle's rotate-half arithmetic. Both take
bf16 roundings at the same points, so they agree to fp64 rounding except where a value
lies within that rounding of a bf16 boundary; the seeded cases below have no such value
(a flip would show as a difference of one bf16 step, far above the 1e-9 checked).
"""
import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import forward as FW
from oracle.retrieval import bf16_to_f64, f32_to_bf16_rne

pytestmark = pytest.mark.filterwarnings("ignore::UserWarning")


def _bits(x):
    return f32_to_bf16_rne(np.asarray(x, dtype=np.float32))


def _weights(rng, D, Hq, Hkv, d, I, bias=True):
    nqkv = (Hq + 2 * Hkv) * d
    return {
        "ln1": _bits(1.0 + 0.1 * rng.standard_normal(D)),
        "wqkv": _bits(rng.standard_normal((nqkv, D)) / np.sqrt(D)),
        "bqkv": _bits(0.1 * rng.standard_normal(nqkv)) if bias else None,
        "wo": _bits(rng.standard_normal((D, Hq * d)) / np.sqrt(Hq * d)),
        "ln2": _bits(1.0 + 0.1 * rng.standard_normal(D)),
        "wgu": _bits(rng.standard_normal((2 * I, D)) / np.sqrt(D)),
        "wd": _bits(rng.standard_normal((D, I)) / np.sqrt(I)),
    }


def _t(bits):
    return torch.from_numpy(bf16_to_f64(bits))


def _bf(x):
    return x.to(torch.bfloat16).to(torch.float64)


def _rope_complex(x, pos, theta):
    """x [R][H][d] torch fp64; pair (j, j + d/2) as the complex number x_j + i x_{j+d/2},
    multiplied by exp(i pos theta^(-2j/d))."""
    d = x.shape[-1]
    half = d // 2
    inv = theta ** (-2.0 * torch.arange(half, dtype=torch.float64) / d)
    ang = pos[:, None].to(torch.float64) * inv[None, :]
    rot = torch.polar(torch.ones_like(ang), ang)[:, None, :]
    z = torch.complex(x[..., :half], x[..., half:]) * rot
    return torch.cat([z.real, z.imag], dim=-1)


def _library_layer(h, w, hist_k, hist_v, Hq, Hkv, pos0, eps, theta):
    """A GQA decoder layer from torch library calls. hist_k/hist_v [Hkv][N][d] fp64."""
    R, D = h.shape
    d = D // Hq
    x = _bf(F.rms_norm(h, (D,), weight=_t(w["ln1"]), eps=eps))
    y = F.linear(x, _t(w["wqkv"]), None if w["bqkv"] is None else _t(w["bqkv"]))
    pos = torch.arange(R) + pos0
    q = _bf(_rope_complex(y[:, :Hq * d].reshape(R, Hq, d), pos, theta))
    k = _bf(_rope_complex(y[:, Hq * d:(Hq + Hkv) * d].reshape(R, Hkv, d), pos, theta))
    v = _bf(y[:, (Hq + Hkv) * d:].reshape(R, Hkv, d))
    N = hist_k.shape[1]
    K = torch.cat([hist_k, k.transpose(0, 1)], dim=1)           # [Hkv][N + R][d]
    V = torch.cat([hist_v, v.transpose(0, 1)], dim=1)
    mask = torch.ones(R, N + R, dtype=torch.bool)
    mask[:, N:] = torch.tril(torch.ones(R, R, dtype=torch.bool))
    o = F.scaled_dot_product_attention(q.transpose(0, 1)[None], K[None], V[None],
                                       attn_mask=mask, enable_gqa=True)[0]  # [Hq][R][d]
    o = _bf(o.transpose(0, 1).reshape(R, Hq * d))
    h1 = h + F.linear(o, _t(w["wo"]))
    x2 = _bf(F.rms_norm(h1, (D,), weight=_t(w["ln2"]), eps=eps))
    I = w["wgu"].shape[0] // 2
    wgu = _t(w["wgu"])
    a = _bf(F.silu(F.linear(x2, wgu[:I])) * F.linear(x2, wgu[I:]))
    h2 = h1 + F.linear(a, _t(w["wd"]))
    return {"h": h2, "q": q, "o": o}


def _compare(ref, lib, atol):
    np.testing.assert_allclose(ref["q"], lib["q"].numpy(), rtol=0, atol=atol)
    np.testing.assert_allclose(ref["o"], lib["o"].numpy(), rtol=0, atol=atol)
    np.testing.assert_allclose(ref["h"], lib["h"].numpy(), rtol=0, atol=atol)


@pytest.mark.parametrize("bias", [True, False])
def test_layer_without_stored_tokens_matches_library_decoder(bias):
    rng = np.random.default_rng(3)
    Hq, Hkv, d, I, R = 4, 2, 8, 24, 5
    D = Hq * d
    w = _weights(rng, D, Hq, Hkv, d, I, bias)
    h = bf16_to_f64(_bits(rng.standard_normal((R, D))))
    empty = np.zeros((Hkv, 0, d), np.uint16)
    ref = FW.layer(h, w, empty, empty, n_q_heads=Hq, n_kv_heads=Hkv, pos0=7, eps=1e-6,
                   theta=1e4)
    lib = _library_layer(torch.from_numpy(h), w, torch.zeros(Hkv, 0, d),
                         torch.zeros(Hkv, 0, d), Hq, Hkv, 7, 1e-6, 1e4)
    _compare(ref, lib, 1e-9)


def test_stored_tokens_match_attention_with_a_prefix_mask():
    rng = np.random.default_rng(5)
    Hq, Hkv, d, I, R, N = 6, 2, 16, 32, 4, 37
    D = Hq * d
    w = _weights(rng, D, Hq, Hkv, d, I)
    h = bf16_to_f64(_bits(rng.standard_normal((R, D))))
    hk = _bits(rng.standard_normal((Hkv, N, d)))
    hv = _bits(rng.standard_normal((Hkv, N, d)))
    ref = FW.layer(h, w, hk, hv, n_q_heads=Hq, n_kv_heads=Hkv, pos0=N, eps=1e-5,
                   theta=1e6)
    lib = _library_layer(torch.from_numpy(h), w, _t(hk), _t(hv), Hq, Hkv, N, 1e-5, 1e6)
    _compare(ref, lib, 1e-9)


def test_attention_alone_against_sdpa_and_uniform_case():
    rng = np.random.default_rng(11)
    R, Hq, Hkv, d, N = 3, 4, 1, 8, 10
    q = rng.standard_normal((R, Hq, d))
    hk, hv = rng.standard_normal((Hkv, N, d)), rng.standard_normal((Hkv, N, d))
    ok, ov = rng.standard_normal((R, Hkv, d)), rng.standard_normal((R, Hkv, d))
    o = FW.attention(q, hk, hv, ok, ov)
    for r in range(R):
        K = np.concatenate([hk, ok[:r + 1].transpose(1, 0, 2)], axis=1)
        V = np.concatenate([hv, ov[:r + 1].transpose(1, 0, 2)], axis=1)
        lib = F.scaled_dot_product_attention(torch.from_numpy(q[r][:, None, :]),
                                             torch.from_numpy(np.repeat(K, Hq, 0)),
                                             torch.from_numpy(np.repeat(V, Hq, 0)))
        np.testing.assert_allclose(o[r], lib[:, 0].numpy(), rtol=0, atol=1e-12)
    # a zero query attends uniformly: the output is the plain mean of the values it sees
    o0 = FW.attention(np.zeros((R, Hq, d)), hk, hv, ok, ov)
    for r in range(R):
        V = np.concatenate([hv[0], ov[:r + 1, 0]], axis=0)
        np.testing.assert_allclose(o0[r], np.broadcast_to(V.mean(0), (Hq, d)), atol=1e-12)


def test_rope_invariants():
    rng = np.random.default_rng(1)
    d, theta = 128, 1e6
    q = rng.standard_normal((1, 1, d))
    k = rng.standard_normal((1, 1, d))
    # identity at position 0, norms kept
    np.testing.assert_allclose(FW.rope(q, np.array([0]), theta), q, atol=0)
    for p in (1, 1000, 705_600):
        np.testing.assert_allclose(np.linalg.norm(FW.rope(q, np.array([p]), theta)),
                                   np.linalg.norm(q), rtol=1e-12)
    # the logit of positions (m, n) depends on m - n only
    for m, n, s in ((5, 2, 11), (700_000, 3, 123_456), (9, 9, 40)):
        a = FW.rope(q, np.array([m]), theta).ravel() @ FW.rope(k, np.array([n]), theta).ravel()
        b = FW.rope(q, np.array([m + s]), theta).ravel() @ FW.rope(k, np.array([n + s]),
                                                                    theta).ravel()
        assert abs(a - b) < 1e-9 * (1 + abs(a))
    # the complex-rotation formulation
    pos = np.array([3, 70_001])
    x = rng.standard_normal((2, 3, d))
    np.testing.assert_allclose(FW.rope(x, pos, theta),
                               _rope_complex(torch.from_numpy(x), torch.from_numpy(pos),
                                             theta).numpy(), atol=1e-12)


def test_rms_norm_closed_form_and_silu_library():
    h = np.full((2, 64), -3.0)
    w = np.linspace(0.5, 1.5, 64)
    np.testing.assert_allclose(FW.rms_norm(h, w, 0.0), -w[None, :].repeat(2, 0), atol=1e-15)
    x = np.linspace(-30, 30, 101)
    np.testing.assert_allclose(FW.silu(x), F.silu(torch.from_numpy(x)).numpy(), atol=1e-15)


def test_zero_weights_leave_the_hidden_states_and_give_rotated_biases():
    rng = np.random.default_rng(2)
    Hq, Hkv, d, I, R, N = 2, 1, 8, 16, 3, 5
    D = Hq * d
    w = _weights(rng, D, Hq, Hkv, d, I)
    for k in ("wqkv", "wo", "wgu", "wd"):
        w[k] = np.zeros_like(w[k])
    h = rng.standard_normal((R, D))
    hk = _bits(rng.standard_normal((Hkv, N, d)))
    r = FW.layer(h, w, hk, hk, n_q_heads=Hq, n_kv_heads=Hkv, pos0=N, eps=1e-6, theta=1e4)
    np.testing.assert_array_equal(r["h"], h)
    b = bf16_to_f64(w["bqkv"])
    q_expect = FW.bf16_round(FW.rope(np.broadcast_to(b[:Hq * d].reshape(1, Hq, d), (R, Hq, d)),
                                     N + np.arange(R), 1e4))
    np.testing.assert_array_equal(r["q"], q_expect)


def test_forward_chains_layers_and_positions_follow_the_stored_tokens():
    rng = np.random.default_rng(4)
    P, Hq, Hkv, d, I, R, N = 2, 4, 2, 8, 16, 3, 9
    D = Hq * d
    layers = [_weights(rng, D, Hq, Hkv, d, I) for _ in range(P)]
    kb = _bits(rng.standard_normal((P, Hkv, N, d)))
    vb = _bits(rng.standard_normal((P, Hkv, N, d)))
    hin = _bits(rng.standard_normal((R, D)))
    out = FW.forward(hin, layers, kb, vb, n_q_heads=Hq, n_kv_heads=Hkv, theta=1e4)
    h = bf16_to_f64(hin)
    for i in range(P):
        lib = _library_layer(torch.from_numpy(h), layers[i], _t(kb[i]), _t(vb[i]), Hq, Hkv,
                             N, 1e-6, 1e4)
        np.testing.assert_allclose(bf16_to_f64(out["q_bits"][i]), lib["q"].numpy(), atol=1e-9)
        h = lib["h"].numpy()
    np.testing.assert_allclose(out["h"], h, atol=1e-9)


def test_planted_mistakes_fail_the_library_comparison(monkeypatch):
    """A sign flip in the rotation or a causal mask off by one must be caught."""
    rng = np.random.default_rng(6)
    Hq, Hkv, d, I, R, N = 4, 2, 8, 16, 4, 6
    D = Hq * d
    w = _weights(rng, D, Hq, Hkv, d, I)
    h = bf16_to_f64(_bits(rng.standard_normal((R, D))))
    hk = _bits(rng.standard_normal((Hkv, N, d)))
    hv = _bits(rng.standard_normal((Hkv, N, d)))
    lib = _library_layer(torch.from_numpy(h), w, _t(hk), _t(hv), Hq, Hkv, N, 1e-6, 1e4)

    def bad_rope(x, pos, theta):
        y = np.asarray(x, np.float64)
        half = y.shape[-1] // 2
        inv = theta ** (-2.0 * np.arange(half) / y.shape[-1])
        ang = np.asarray(pos, np.float64)[:, None] * inv[None, :]
        c, s = np.cos(ang)[:, None], np.sin(ang)[:, None]
        a, b = y[..., :half], y[..., half:]
        return np.concatenate([a * c + b * s, b * c - a * s], axis=-1)    # wrong sense

    for name, fn in (("rope", bad_rope),):
        with monkeypatch.context() as m:
            m.setattr(FW, name, fn)
            bad = FW.layer(h, w, hk, hv, n_q_heads=Hq, n_kv_heads=Hkv, pos0=N, eps=1e-6,
                           theta=1e4)
            assert np.abs(bad["q"] - lib["q"].numpy()).max() > 1e-3

    def shifted_attention(q, hist_k, hist_v, own_k, own_v, spread=False):
        # rows r >= 1 see one own row too few (a causal mask off by one)
        R_, Hq_, d_ = q.shape
        G_ = Hq_ // hist_k.shape[0]
        out = np.zeros_like(q)
        for hh in range(Hq_):
            g = hh // G_
            for r in range(R_):
                lim = max(r, 1)
                K = np.concatenate([hist_k[g], own_k[:lim, g]], axis=0)
                V = np.concatenate([hist_v[g], own_v[:lim, g]], axis=0)
                s_ = K @ q[r, hh] / np.sqrt(d_)
                p_ = np.exp(s_ - s_.max())
                out[r, hh] = (p_ / p_.sum()) @ V
        return out

    with monkeypatch.context() as m:
        m.setattr(FW, "attention", shifted_attention)
        bad = FW.layer(h, w, hk, hv, n_q_heads=Hq, n_kv_heads=Hkv, pos0=N, eps=1e-6,
                       theta=1e4)
        assert np.abs(bad["o"] - lib["o"].numpy()).max() > 1e-3


def test_spread_upper_bound_holds():
    rng = np.random.default_rng(8)
    R, Hq, Hkv, d, N = 4, 4, 2, 8, 50
    q = rng.standard_normal((R, Hq, d))
    hk, hv = rng.standard_normal((Hkv, N, d)), rng.standard_normal((Hkv, N, d))
    ok, ov = rng.standard_normal((R, Hkv, d)), rng.standard_normal((R, Hkv, d))
    o1, exact = FW.attention(q, hk, hv, ok, ov, spread=True)
    o2, upper = FW.attention(q, hk, hv, ok, ov, spread="upper")
    np.testing.assert_array_equal(o1, o2)
    assert (upper >= exact - 1e-12).all() and (exact > 0).all()
