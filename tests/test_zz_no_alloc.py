"""The allocation-free attention entry point (needs a GPU).

ee_attention_decode_static serves callers that cannot allocate device memory
(their HBM belongs to another allocator's pool, their hot path must not call
cudaMalloc, or they have no allocator).  Its scratch is a fixed area inside
the library shared by all calls, so this checks it against the allocating
ee_attention_decode on two calls in a row with different shapes and data
(stale contents of the shared area must not leak from one call into the
next), and that shapes too large for the area are refused.  Collected last so
that a failure here never hides the other tests."""
import ctypes

import numpy as np
import pytest

import oracle
import synth
from helpers import rel_err, to_bf16_bits

pytestmark = pytest.mark.gpu


def _dev(a):
    import torch
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        a = a.view(np.int16)
    return torch.from_numpy(a).cuda()


def _case(seed, T, A, KH, D, P=64):
    rng = np.random.default_rng(seed)
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
    return q, K, V, kp, vp, perm


def test_static_scratch_attention_matches_the_allocating_entry_point():
    import torch

    from paper_2609_14144_gb300 import _lib, attention_decode

    lib = _lib.load()
    stream = torch.cuda.current_stream()
    for seed, (T, A, KH, D) in enumerate([(1000, 12, 2, 128), (77, 14, 2, 64)]):
        q, K, V, kp, vp, perm = _case(seed, T, A, KH, D)
        dq, dk, dv, dp = _dev(q), _dev(kp), _dev(vp), _dev(perm)
        ref = attention_decode(dq, dk, dv, dp, T, A, KH, D, 64)
        out = torch.full((A * D,), float("nan"), dtype=torch.float32, device="cuda")
        rc = lib.ee_attention_decode_static(dq.data_ptr(), dk.data_ptr(), dv.data_ptr(), dp.data_ptr(), T, A, KH, D,
                                            64, out.data_ptr(), ctypes.c_void_p(stream.cuda_stream))
        assert rc == 0, lib.ee_last_error()
        torch.cuda.synchronize()
        got, want = out.cpu().numpy().reshape(A, D), ref.cpu().numpy().reshape(A, D)
        assert np.isfinite(got).all()
        for h in range(A):
            assert rel_err(got[h], want[h]) <= 1e-4, (seed, h)
            g = h // (A // KH)
            expect = oracle.attention(q[h * D:(h + 1) * D], synth.bf16_to_f32(K)[:, g], synth.bf16_to_f32(V)[:, g])
            assert rel_err(got[h], expect) <= 1e-4, (seed, h)


def test_static_scratch_rejects_shapes_beyond_its_size():
    import torch

    from paper_2609_14144_gb300 import _lib

    lib = _lib.load()
    q = torch.zeros(64 * 128, dtype=torch.float32, device="cuda")
    kv = torch.zeros(64 * 128, dtype=torch.int16, device="cuda")
    pt = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = torch.zeros(64 * 128, dtype=torch.float32, device="cuda")
    rc = lib.ee_attention_decode_static(q.data_ptr(), kv.data_ptr(), kv.data_ptr(), pt.data_ptr(), 1, 64, 8, 128, 64,
                                        out.data_ptr(), None)
    assert rc == _lib.EE_EINVAL
    assert b"static area" in lib.ee_last_error()
