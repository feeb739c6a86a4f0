"""Pins of the oracle's vision-transformer operators against closed forms,
textbook constants, invariants and brute force (no GPU)."""
import math

import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2511_19457_gb300 import synth


def _bits(a):
    return synth.to_bf16_bits(torch.as_tensor(np.asarray(a, dtype=np.float32)))


def test_gelu_constants_and_identities():
    # Phi(1) = 0.8413447460685429 (standard normal CDF, tables)
    assert orc.gelu(1.0) == pytest.approx(0.8413447460685429, abs=1e-15)
    assert orc.gelu(0.0) == 0.0
    x = np.linspace(-6, 6, 97)
    # GELU(x) - GELU(-x) = x (Phi(x) + Phi(-x) = 1)
    assert np.allclose(orc.gelu(x) - orc.gelu(-x), x, atol=1e-14)
    assert orc.gelu(8.0) == pytest.approx(8.0, abs=1e-12)
    assert abs(orc.gelu(-8.0)) < 1e-13


def test_gelu_through_the_fc_epilogue():
    """act = 3 in the C epilogue equals x * Phi(x) (computed here with math.erf)."""
    rng = np.random.default_rng(0)
    xb = _bits(rng.standard_normal((3, 8)))
    wb = _bits(np.eye(8))
    y = orc.fc(xb, 3, 8, wb, 8, act=orc.ACT_GELU)
    xv = orc.bf16_to_f64(xb).reshape(3, 8)
    want = np.array([[v * 0.5 * (1 + math.erf(v / math.sqrt(2))) for v in row] for row in xv])
    assert np.allclose(y, want, atol=1e-14)


def test_layernorm_hand_example():
    # x = 1, 2, 3, 4: mean 2.5, biased variance 1.25
    y = orc.layernorm(_bits([[1, 2, 3, 4]]), 1, 4, eps=0.0)
    assert np.allclose(y, (np.array([1, 2, 3, 4]) - 2.5) / math.sqrt(1.25), atol=1e-15)
    gb = np.array([[2, 2, 2, 2], [1, 1, 1, 1]], dtype=np.float32)
    y2 = orc.layernorm(_bits([[1, 2, 3, 4]]), 1, 4, gamma_beta=gb, eps=0.0)
    assert np.allclose(y2, 2 * y + 1, atol=1e-15)


def test_layernorm_moments_and_constant_rows():
    rng = np.random.default_rng(1)
    xb = _bits(3 + 2 * rng.standard_normal((5, 768)))
    eps = 1e-6
    y = orc.layernorm(xb, 5, 768, eps=eps)
    x = orc.bf16_to_f64(xb).reshape(5, 768)
    var = x.var(axis=1)
    assert np.allclose(y.mean(axis=1), 0.0, atol=1e-12)
    assert np.allclose(y.var(axis=1), var / (var + eps), atol=1e-12)  # closed form
    assert np.all(orc.layernorm(_bits(np.full((2, 16), 3.5)), 2, 16) == 0.0)


def _attention_brute(q, k, v):
    """Pure-Python loops: softmax over keys of the scaled dot products."""
    T, hd = q.shape
    out = np.zeros_like(q)
    for t in range(T):
        s = [sum(q[t, d] * k[j, d] for d in range(hd)) / math.sqrt(hd) for j in range(T)]
        m = max(s)
        e = [math.exp(x - m) for x in s]
        z = sum(e)
        for d in range(hd):
            out[t, d] = sum(e[j] / z * v[j, d] for j in range(T))
    return out


def test_attention_brute_force_tiny():
    rng = np.random.default_rng(2)
    N, T, H, hd = 2, 3, 2, 4
    qkv = rng.standard_normal((N, T, 3 * H * hd))
    xb = _bits(qkv)
    y = orc.attention(xb, N, T, H, hd)
    x = orc.bf16_to_f64(xb).reshape(N, T, 3, H, hd)
    for n in range(N):
        for h in range(H):
            want = _attention_brute(x[n, :, 0, h], x[n, :, 1, h], x[n, :, 2, h])
            assert np.allclose(y[n, :, h * hd:(h + 1) * hd], want, atol=1e-13)


def test_attention_invariants():
    rng = np.random.default_rng(3)
    N, T, H, hd = 1, 6, 2, 8
    x = rng.standard_normal((N, T, 3, H, hd))
    # identical keys: uniform weights, every output row is the mean of V
    x[:, :, 1] = x[:, :1, 1]
    y = orc.attention(_bits(x.reshape(N, T, -1)), N, T, H, hd)
    v = orc.bf16_to_f64(_bits(x.reshape(N, T, -1))).reshape(N, T, 3, H, hd)[:, :, 2]
    assert np.allclose(y.reshape(N, T, H, hd), v.mean(axis=1, keepdims=True), atol=1e-13)
    # permuting the tokens permutes the output rows the same way
    x2 = rng.standard_normal((N, T, 3 * H * hd))
    perm = rng.permutation(T)
    y2 = orc.attention(_bits(x2), N, T, H, hd)
    y2p = orc.attention(_bits(x2[:, perm]), N, T, H, hd)
    assert np.allclose(y2p, y2[:, perm], atol=1e-13)


def test_tokens_and_select():
    rng = np.random.default_rng(4)
    N, P, D = 2, 4, 8
    x = rng.standard_normal((N, P, D))
    cls = rng.standard_normal(D)
    pos = rng.standard_normal((P + 1, D)).astype(np.float32)
    seq = orc.tokens(_bits(x), N, P, D, _bits(cls), pos)
    xb = orc.bf16_to_f64(_bits(x)).reshape(N, P, D)
    cb = orc.bf16_to_f64(_bits(cls))
    assert np.array_equal(seq[:, 0], np.broadcast_to(cb + pos[0].astype(np.float64), (N, D)))
    assert np.array_equal(seq[:, 1:], xb + pos[1:].astype(np.float64))
    s = orc.select_token(_bits(seq), N, P + 1, D, 0)
    assert np.array_equal(s, orc.bf16_to_f64(_bits(seq)).reshape(N, P + 1, D)[:, 0])


def test_vit_b16_macs_table2():
    """ViT-B16 is quoted at 17.6 G (Table 2): patch embedding, 12 encoder
    layers (QKV, Q K^T, P V, projection, MLP 768-3072-768) and the head."""
    T, D, Hm = 197, 768, 3072
    patch = 196 * 768 * (16 * 16 * 3)
    layer = T * D * 3 * D + 2 * T * T * D + T * D * D + 2 * T * D * Hm
    macs = patch + 12 * layer + D * 1000
    assert 17.5e9 < macs < 17.65e9
    ops, _, shape = synth.vit(batch=1)
    got = synth_macs(ops, shape)
    assert got == macs


def synth_macs(ops, shape):
    """MACs of a ViT operator list from its shapes (patch embedding on the
    real 3 input channels, as Table 2 counts it)."""
    from paper_2511_19457_gb300 import calibrate as cal
    ins = cal.graph_input_shapes(ops, shape)
    macs = 0
    for op, (B, H, W, C) in zip(ops, ins):
        if op["kind"] == "conv":
            Ho = (H + 2 * op["pad"] - op["k"]) // op["stride"] + 1
            Wo = (W + 2 * op["pad"] - op["k"]) // op["stride"] + 1
            macs += B * Ho * Wo * op["cout"] * C * op["k"] * op["k"]
        elif op["kind"] == "fc":
            macs += B * H * W * C * op["cout"]
        elif op["kind"] == "attention":
            T = H * W
            D = C // 3
            macs += 2 * B * T * T * D
    return macs
