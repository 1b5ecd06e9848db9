"""Shared helpers for the test suite: small model shapes and weight edits."""
from __future__ import annotations

import numpy as np
import torch

import synth


def micro(**kw) -> synth.ModelShape:
    """A few-layer decoder small enough for brute-force checks."""
    base = dict(name="micro", n_layers=4, d_model=64, n_heads=4, n_kv_heads=2, head_dim=16, ffn_dim=96,
                vocab=300, readout_layers=(2,), seed=7, prompt_len=8, new_tokens=8)
    base.update(kw)
    return synth.ModelShape(**base)


def to_bf16_bits(a) -> np.ndarray:
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16).copy()


def bf16_round(a) -> np.ndarray:
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16).float().numpy()


def zeros_like_bits(a) -> np.ndarray:
    return np.zeros_like(np.asarray(a, dtype=np.uint16))


def one_hot_matrix(rows: int, cols: int, i: int, j: int, value: float = 1.0) -> np.ndarray:
    m = np.zeros((rows, cols), np.float32)
    m[i, j] = value
    return to_bf16_bits(m)


def identity_bits(n: int) -> np.ndarray:
    return to_bf16_bits(np.eye(n, dtype=np.float32))
