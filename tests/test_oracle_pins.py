"""Pins of the oracle's ops against closed forms, library routines and brute
force (no GPU).  Each op is checked by something other than itself, chosen so
that a dropped term, a wrong sign or index, or a transposed operand fails."""
import math

import numpy as np
import pytest
import scipy.special
import scipy.stats
import torch

import oracle
import synth

RNG = np.random.default_rng(1234)


# ------------------------------------------------------------- bf16 rounding
def test_bf16_round_matches_torch_rne():
    x = np.concatenate([
        RNG.standard_normal(20000).astype(np.float32) * 10.0 ** RNG.integers(-30, 30, 20000),
        # exact halfway cases: lower 16 bits 0x8000 with odd and even kept lsb
        (np.arange(1000, dtype=np.uint32) << 16 | 0x8000).view(np.float32),
        (np.arange(1000, dtype=np.uint32) << 16 | 0x7FFF).view(np.float32),
        np.array([0.0, -0.0, 1e-40, -1e-40, 3.4e38, -3.4e38, np.inf, -np.inf], dtype=np.float32),
    ]).astype(np.float32)
    ours = oracle.bf16_round(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float32).numpy()
    assert np.array_equal(ours.view(np.uint32), ref.view(np.uint32))
    assert np.isnan(oracle.bf16_round(np.array([np.nan], np.float32))[0])


def test_bf16_round_ties_to_even_by_hand():
    # 1 + 2^-8 lies halfway between bf16 1.0 and 1 + 2^-7; even mantissa is 1.0
    assert oracle.bf16_round(np.float32(1 + 2 ** -8))[0] == 1.0
    # 1 + 3 * 2^-8 lies halfway between 1 + 2^-7 (odd) and 1 + 2^-6 (even)
    assert oracle.bf16_round(np.float32(1 + 3 * 2 ** -8))[0] == np.float32(1 + 2 ** -6)


# ------------------------------------------------------------- matvec
def _to_bf16_bits(a: np.ndarray) -> np.ndarray:
    return torch.from_numpy(np.asarray(a, np.float32)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def test_matvec_exact_on_small_integers():
    W = RNG.integers(-8, 9, size=(37, 301)).astype(np.float32)
    b = RNG.integers(-8, 9, size=37).astype(np.float32)
    x = RNG.integers(-8, 9, size=301).astype(np.float32)
    out = oracle.matvec(_to_bf16_bits(W), x, _to_bf16_bits(b))
    exact = W.astype(np.int64) @ x.astype(np.int64) + b.astype(np.int64)
    assert np.array_equal(out.astype(np.int64), exact)


def test_matvec_orientation_and_values_against_numpy():
    W = RNG.standard_normal((53, 200)).astype(np.float32) * 0.05
    Wb = _to_bf16_bits(W)
    x = RNG.standard_normal(200).astype(np.float32)
    out = oracle.matvec(Wb, x)
    ref = synth.bf16_to_f32(Wb).astype(np.float64) @ x.astype(np.float64)
    assert out.shape == (53,)
    np.testing.assert_allclose(out, ref, rtol=1e-6, atol=1e-7)


# ------------------------------------------------------------- RMSNorm
def test_rmsnorm_constant_vector_closed_form():
    d, c, eps = 64, 0.37, 1e-6
    g = _to_bf16_bits(np.linspace(-2, 2, d))
    out = oracle.rmsnorm(np.full(d, c, np.float32), g, eps)
    expect = synth.bf16_to_f32(g).astype(np.float64) * c / math.sqrt(c * c + eps)
    np.testing.assert_allclose(out, expect, rtol=1e-6)


def test_rmsnorm_unit_rms_and_scale_invariance():
    d = 300
    h = RNG.standard_normal(d).astype(np.float32) * 3
    ones = synth.const_bf16(d, 1.0)
    u = oracle.rmsnorm(h, ones, 0.0)
    assert np.sqrt(np.mean(u.astype(np.float64) ** 2)) == pytest.approx(1.0, rel=1e-6)
    u2 = oracle.rmsnorm(h * np.float32(8.0), ones, 0.0)
    np.testing.assert_allclose(u2, u, rtol=1e-6)
    # the gain multiplies element-wise
    two = synth.const_bf16(d, 2.0)
    np.testing.assert_array_equal(oracle.rmsnorm(h, two, 0.0), 2 * u)


# ------------------------------------------------------------- RoPE
def test_rope_identity_at_position_zero():
    x = RNG.standard_normal(128).astype(np.float32)
    assert np.array_equal(oracle.rope(x, 0, 10000.0), x)


def test_rope_single_pair_is_rotation_by_position():
    for t in (1, 2, 7, 1000):
        out = oracle.rope(np.array([1.0, 0.0], np.float32), t, 10000.0)
        np.testing.assert_allclose(out, [math.cos(t), math.sin(t)], atol=1e-6)


def test_rope_rotate_half_pairing_and_frequency():
    # D = 4: pairs (0, 2) at frequency 1 and (1, 3) at base^(-1/2)
    base, t = 10000.0, 3
    e0 = oracle.rope(np.array([1, 0, 0, 0], np.float32), t, base)
    np.testing.assert_allclose(e0, [math.cos(t), 0, math.sin(t), 0], atol=1e-6)
    e1 = oracle.rope(np.array([0, 1, 0, 0], np.float32), t, base)
    w = t * base ** -0.5
    np.testing.assert_allclose(e1, [0, math.cos(w), 0, math.sin(w)], atol=1e-6)
    e3 = oracle.rope(np.array([0, 0, 0, 1], np.float32), t, base)
    np.testing.assert_allclose(e3, [0, -math.sin(w), 0, math.cos(w)], atol=1e-6)


def test_rope_preserves_pair_norms_and_scores_depend_on_offset_only():
    D = 128
    q = RNG.standard_normal(D).astype(np.float32)
    k = RNG.standard_normal(D).astype(np.float32)
    for t in (5, 4096):
        r = oracle.rope(q, t, 10000.0).astype(np.float64)
        n_in = q[:64].astype(np.float64) ** 2 + q[64:].astype(np.float64) ** 2
        n_out = r[:64] ** 2 + r[64:] ** 2
        np.testing.assert_allclose(n_out, n_in, rtol=1e-5)
    ref = float(oracle.rope(q, 10, 1e4).astype(np.float64) @ oracle.rope(k, 3, 1e4).astype(np.float64))
    for shift in (0, 1, 4096):
        s = float(oracle.rope(q, 10 + shift, 1e4).astype(np.float64) @ oracle.rope(k, 3 + shift, 1e4).astype(np.float64))
        assert s == pytest.approx(ref, rel=2e-4, abs=2e-4)


# ------------------------------------------------------------- attention
@pytest.mark.parametrize("T", [1, 2, 15, 16, 17, 63, 64, 65])
@pytest.mark.parametrize("D", [64, 128])
def test_attention_brute_force(T, D):
    q = RNG.standard_normal(D).astype(np.float32)
    K = RNG.standard_normal((T, D)).astype(np.float32)
    V = RNG.standard_normal((T, D)).astype(np.float32)
    out = oracle.attention(q, K, V)
    p = scipy.special.softmax(K.astype(np.float64) @ q.astype(np.float64) / math.sqrt(D))
    np.testing.assert_allclose(out, p @ V.astype(np.float64), rtol=1e-5, atol=1e-6)


def test_attention_special_cases():
    D = 64
    V = RNG.standard_normal((9, D)).astype(np.float32)
    q = RNG.standard_normal(D).astype(np.float32)
    # one position: the output is that value row
    np.testing.assert_array_equal(oracle.attention(q, V[:1] * 0 + 1, V[:1]), V[0])
    # identical keys: uniform weights, the output is the mean of the values
    K = np.tile(RNG.standard_normal(D).astype(np.float32), (9, 1))
    np.testing.assert_allclose(oracle.attention(q, K, V), V.astype(np.float64).mean(0), rtol=1e-5, atol=1e-6)
    # one key aligned with a large query: the output is that key's value
    K = np.zeros((9, D), np.float32)
    K[4] = q * 50
    np.testing.assert_allclose(oracle.attention(q, K, V), V[4], rtol=1e-5, atol=1e-5)


# ------------------------------------------------------------- SiLU
def test_silu_closed_forms():
    x = np.linspace(-30, 30, 1001)
    s = oracle.silu(x)
    assert oracle.silu(np.array([0.0]))[0] == 0.0
    np.testing.assert_allclose(s - oracle.silu(-x), x, atol=1e-12)
    np.testing.assert_allclose(s, x * scipy.special.expit(x), rtol=1e-13, atol=1e-300)


# ------------------------------------------------------------- confidence
def test_confidence_against_logsumexp():
    for V in (2, 17, 4096, 151936):
        l = (RNG.standard_normal(V) * 7).astype(np.float32)
        c = oracle.confidence(l)
        lse = scipy.special.logsumexp(l.astype(np.float64))
        assert c["argmax"] == int(np.argmax(l))
        assert c["p1"] == pytest.approx(math.exp(float(l.max()) - lse), rel=1e-6)
        second = np.sort(l)[-2]
        assert c["p2"] == pytest.approx(math.exp(float(second) - lse), rel=1e-6)
        assert 1.0 / V <= c["p1"] <= 1.0


def test_confidence_special_cases():
    V = 1000
    c = oracle.confidence(np.zeros(V, np.float32))
    assert c["p1"] == pytest.approx(1.0 / V, rel=1e-6) and c["argmax"] == 0 and c["gap"] == 0.0
    l = np.zeros(V, np.float32)
    l[321] = 100.0
    c = oracle.confidence(l)
    assert c["argmax"] == 321 and c["p1"] == pytest.approx(1.0, abs=1e-30 + 1e-6)
    # ties resolve to the lowest index
    l = RNG.standard_normal(V).astype(np.float32)
    l[[10, 500, 900]] = 9.0
    c = oracle.confidence(l)
    assert c["argmax"] == 10 and c["gap"] == 0.0
    # two logits: p1 = 1 / (1 + exp(b - a))
    c = oracle.confidence(np.array([1.5, 0.25], np.float32))
    assert c["p1"] == pytest.approx(1 / (1 + math.exp(-1.25)), rel=1e-7)
    assert c["gap"] == pytest.approx(c["p1"] - (1 - c["p1"]), rel=1e-6)


def test_negative_entropy_and_margin_against_scipy():
    """Section 10's other two signals: margin p1 - p2 and negative entropy
    sum p log p, against scipy's entropy and a sorted softmax."""
    for V in (2, 17, 4096, 151936):
        l = (RNG.standard_normal(V) * 5).astype(np.float32)
        c = oracle.confidence(l)
        p = scipy.special.softmax(l.astype(np.float64))
        assert c["neg_entropy"] == pytest.approx(-scipy.stats.entropy(p), rel=1e-6, abs=1e-7)
        top = np.sort(p)[-2:]
        assert c["gap"] == pytest.approx(top[1] - top[0], rel=1e-5, abs=1e-7)


def test_negative_entropy_and_margin_closed_forms():
    V = 1000
    c = oracle.confidence(np.zeros(V, np.float32))  # uniform: -log V, no margin
    assert c["neg_entropy"] == pytest.approx(-math.log(V), rel=1e-6) and c["gap"] == 0.0
    # one logit a above V - 1 equal ones: p1 = e^a / (e^a + V - 1), the rest q
    a = 4.0
    l = np.zeros(V, np.float32)
    l[7] = a
    c = oracle.confidence(l)
    z = math.exp(a) + V - 1
    p1, q = math.exp(a) / z, 1.0 / z
    assert c["neg_entropy"] == pytest.approx(p1 * math.log(p1) + (V - 1) * q * math.log(q), rel=1e-6)
    assert c["gap"] == pytest.approx(p1 - q, rel=1e-6)
    # near one-hot: negative entropy tends to 0 from below
    l[7] = 60.0
    c = oracle.confidence(l)
    assert -1e-20 < -c["neg_entropy"] < 1e-20 + 1e-12 and c["neg_entropy"] <= 0.0
    # two logits: -H = p log p + (1 - p) log(1 - p)
    c = oracle.confidence(np.array([0.5, -0.75], np.float32))
    p = 1 / (1 + math.exp(-1.25))
    assert c["neg_entropy"] == pytest.approx(p * math.log(p) + (1 - p) * math.log(1 - p), rel=1e-6)


def _nucleus_by_sorting(l, x, p_nuc):
    """The nucleus as the smallest set of most probable tokens whose
    probability reaches p_nuc, by sorting (continuous logits, no ties)."""
    p = scipy.special.softmax(l.astype(np.float64))
    order = np.argsort(-p, kind="stable")
    k = int(np.searchsorted(np.cumsum(p[order]), p_nuc)) + 1
    return x in set(order[:k].tolist())


def test_nucleus_membership_against_sorting():
    """Section 2: a token is in the nucleus when it belongs to the smallest
    set of most probable tokens holding 90 percent of the probability."""
    for V, scale in ((50, 1.0), (4096, 3.0), (151936, 6.0)):
        l = (RNG.standard_normal(V) * scale).astype(np.float32)
        order = np.argsort(-l)
        for x in list(order[:40]) + list(RNG.integers(0, V, 20)):
            got, mass = oracle.nucleus_member(l, int(x), 0.9)
            assert got == _nucleus_by_sorting(l, int(x), 0.9), (V, x, mass)
            p = scipy.special.softmax(l.astype(np.float64))
            assert mass == pytest.approx(float(p[p > p[x]].sum()), rel=1e-9, abs=1e-12)


def test_nucleus_membership_special_cases():
    V = 1000
    # uniform: nothing is more probable than any token, all are members
    assert all(oracle.nucleus_member(np.zeros(V, np.float32), x)[0] for x in (0, 499, 999))
    # one token holding more than 90 percent: the nucleus is that token alone
    l = np.zeros(V, np.float32)
    l[5] = 20.0
    assert oracle.nucleus_member(l, 5)[0] and not oracle.nucleus_member(l, 6)[0]
    # share 1.0 keeps every token
    l = (RNG.standard_normal(V) * 4).astype(np.float32)
    assert all(oracle.nucleus_member(l, x, 1.0)[0] for x in range(0, V, 97))


def _select_tau_brute(conf, member, target):
    best = math.inf
    for cand in [-math.inf] + sorted(set(float(c) for c in conf)):
        early = [m for c, m in zip(conf, member) if c > cand]
        if early and sum(early) >= target * len(early):
            best = min(best, cand)
    return best


def test_select_tau_against_brute_force():
    """Section 4, step four: the lowest threshold at which the required share
    of early answers is acceptable."""
    for n, q in ((1, 0.5), (7, 0.5), (200, 0.8), (2000, 0.6)):
        conf = RNG.random(n).astype(np.float32)
        member = (RNG.random(n) < q * (0.5 + conf)).astype(np.int32)
        for target in (0.5, 0.9, 0.99):
            assert oracle.select_tau(conf, member, target) == np.float32(_select_tau_brute(conf, member, target))
    # every answer acceptable: everything may exit; none acceptable: nothing may
    conf = RNG.random(50).astype(np.float32)
    assert oracle.select_tau(conf, np.ones(50, np.int32), 0.9) == -math.inf
    assert oracle.select_tau(conf, np.zeros(50, np.int32), 0.9) == math.inf
    # acceptability rising with confidence: tau sits just below the good run
    conf = np.arange(10, dtype=np.float32) / 10
    member = np.array([0, 0, 0, 1, 0, 1, 1, 1, 1, 1], np.int32)
    assert oracle.select_tau(conf, member, 1.0) == np.float32(0.4)
    assert oracle.select_tau(conf, member, 0.8) == np.float32(0.2)
