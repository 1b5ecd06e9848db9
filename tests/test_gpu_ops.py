"""Standalone kernels through the C ABI vs the oracle's ops (needs a GB300).

Split-K paged attention over T in {1, 2, 15, 16, 17, 63, 64, 65, 1000, 8192}
and several head groupings; the vocabulary pass with ragged vocabularies."""
import math

import numpy as np
import pytest

import oracle
import synth
from helpers import rel_err, to_bf16_bits

pytestmark = pytest.mark.gpu


def _dev(a, dtype=None):
    """numpy -> CUDA tensor; 16-bit bit patterns travel as int16."""
    import torch
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        a = a.view(np.int16)
    return torch.from_numpy(a).cuda()


@pytest.mark.parametrize("T", [1, 2, 15, 16, 17, 63, 64, 65, 1000, 8192])
@pytest.mark.parametrize("A,KH,D", [(12, 2, 128), (14, 2, 64), (4, 2, 64), (16, 2, 128), (8, 8, 64)])
def test_attention_decode(T, A, KH, D):
    import torch

    from paper_2609_14144_gb300 import attention_decode

    rng = np.random.default_rng(T * 31 + A)
    P = 64
    n_pages = (T + P - 1) // P
    perm = rng.permutation(n_pages).astype(np.int32)
    q = rng.standard_normal(A * D).astype(np.float32)
    K = to_bf16_bits(rng.standard_normal((T, KH, D)).astype(np.float32))
    V = to_bf16_bits(rng.standard_normal((T, KH, D)).astype(np.float32))
    kp = np.zeros((n_pages, KH, P, D), np.uint16)
    vp = np.zeros((n_pages, KH, P, D), np.uint16)
    for t in range(T):
        kp[perm[t // P], :, t % P] = K[t]
        vp[perm[t // P], :, t % P] = V[t]
    out = attention_decode(_dev(q), _dev(kp), _dev(vp), _dev(perm), T, A, KH, D, P)
    torch.cuda.synchronize()
    got = out.cpu().numpy().reshape(A, D)
    Kf, Vf = synth.bf16_to_f32(K), synth.bf16_to_f32(V)
    for h in range(A):
        g = h // (A // KH)
        ref = oracle.attention(q[h * D:(h + 1) * D], Kf[:, g], Vf[:, g])
        assert rel_err(got[h], ref) <= 1e-4, (h, rel_err(got[h], ref))


@pytest.mark.parametrize("V,d", [(4096, 256), (4093, 256), (151936, 896), (151937, 1536), (1000, 2048)])
def test_vocab_confidence(V, d):
    import torch

    from paper_2609_14144_gb300 import vocab_confidence

    rng = np.random.default_rng(V + d)
    x = rng.standard_normal(d).astype(np.float32)
    gain = synth.const_bf16(d, 7.0 / (0.02 * math.sqrt(d)))
    U = synth.normal_bf16(5, 0x777, (V, d))
    logits = torch.empty(V, dtype=torch.float32, device="cuda")
    tok, p = vocab_confidence(_dev(x), _dev(gain), _dev(U), 1e-6, logits=logits)
    torch.cuda.synchronize()
    z = oracle.rmsnorm(x, gain, 1e-6)
    ref_l = oracle.matvec(U, z)
    c = oracle.confidence(ref_l)
    assert rel_err(logits.cpu().numpy(), ref_l) <= 1e-4
    assert abs(float(p.item()) - c["p1"]) <= 1e-4
    if c["gap"] >= 1e-3:
        assert int(tok.item()) == c["argmax"]


@pytest.mark.parametrize("V,d", [(4096, 256), (151936, 1536), (1000, 2048)])
def test_vocab_signals(V, d):
    """Section 10's three signals from one pass, against the oracle's
    definitions on the same logits."""
    import torch

    from paper_2609_14144_gb300 import vocab_signals

    rng = np.random.default_rng(V * 3 + d)
    x = rng.standard_normal(d).astype(np.float32)
    gain = synth.const_bf16(d, 4.0 / (0.02 * math.sqrt(d)))
    U = synth.normal_bf16(6, 0x778, (V, d))
    tok, sig = vocab_signals(_dev(x), _dev(gain), _dev(U), 1e-6)
    torch.cuda.synchronize()
    c = oracle.confidence(oracle.matvec(U, oracle.rmsnorm(x, gain, 1e-6)))
    got = sig.cpu().numpy()
    assert abs(got[0] - c["p1"]) <= 1e-4
    assert abs(got[1] - c["gap"]) <= 1e-4
    assert abs(got[2] - c["neg_entropy"]) <= 1e-4 * max(1.0, abs(c["neg_entropy"]))
    if c["gap"] >= 1e-3:
        assert int(tok.item()) == c["argmax"]


def test_vocab_signals_tie_and_uniform():
    import torch

    from paper_2609_14144_gb300 import vocab_signals

    V, d = 50000, 256
    U = np.zeros((V, d), np.uint16)
    row = to_bf16_bits(np.linspace(-1, 1, d).astype(np.float32))
    for v in (40000, 12345, 49999):
        U[v] = row
    x = np.linspace(-1, 1, d).astype(np.float32)
    gain = synth.const_bf16(d, 1.0)
    tok, sig = vocab_signals(_dev(x), _dev(gain), _dev(U), 1e-6)
    torch.cuda.synchronize()
    c = oracle.confidence(oracle.matvec(U, oracle.rmsnorm(x, gain, 1e-6)))
    assert int(tok.item()) == 12345 and float(sig[1].item()) == 0.0
    assert abs(float(sig[2].item()) - c["neg_entropy"]) <= 1e-4 * abs(c["neg_entropy"])
    # all-zero matrix: uniform distribution, p1 = 1/V, margin 0, -log V
    tok, sig = vocab_signals(_dev(x), _dev(gain), _dev(np.zeros((V, d), np.uint16)), 1e-6)
    torch.cuda.synchronize()
    got = sig.cpu().numpy()
    assert int(tok.item()) == 0 and got[1] == 0.0
    assert abs(got[0] - 1.0 / V) <= 1e-9 and abs(got[2] + math.log(V)) <= 1e-4


def test_vocab_confidence_ties_lowest_index():
    import torch

    from paper_2609_14144_gb300 import vocab_confidence

    V, d = 50000, 256
    U = np.zeros((V, d), np.uint16)
    row = to_bf16_bits(np.linspace(-1, 1, d).astype(np.float32))
    for v in (40000, 12345, 49999):
        U[v] = row
    x = np.linspace(-1, 1, d).astype(np.float32)
    gain = synth.const_bf16(d, 1.0)
    tok, p = vocab_confidence(_dev(x), _dev(gain), _dev(U), 1e-6)
    torch.cuda.synchronize()
    assert int(tok.item()) == 12345
