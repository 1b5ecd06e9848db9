"""Seeded synthetic workloads for the early-exit decode path.

Input data only: model shapes, bf16 weights, readouts, prompts and token
streams, produced from named SplitMix64 streams (see ``synth.c``).  Nothing
here computes any part of the decode method; the CPU oracle and the CUDA
library both consume these arrays.

Weight recipe (all tensors bf16, row-major ``[out, in]``):

* every projection, the embedding and the (untied) LM head: N(0, 0.02^2);
* attention / MLP RMSNorm gains: 1.0;
* final RMSNorm gain: ``s / (0.02 * sqrt(d))`` with ``s = 1.5 * sqrt(2 ln V)``,
  which gives the unembedding's logits a standard deviation of about ``s``
  so that top-1 probabilities spread over (0, 1) instead of sitting near 1/V;
* readout at a layer: ``I + N(0, 0.02^2)`` and offset ``N(0, 0.02^2)``
  (a fitted readout starts at identity and zero, Appendix B).

Stream ids: layer ``j`` (0-based) tensor kind ``k`` uses ``0x1000 + 16*j + k``
with kinds Wq=0, Wk=1, Wv=2, Wo=3, Wg=4, Wu=5, Wd=6, bq=7, bk=8, bv=9; the
embedding uses 0x100, an untied LM head 0x101, readout ``r`` uses
``0x200 + 2r`` (matrix) and ``0x201 + 2r`` (offset), the prompt 0x300, the
calibration stream 0x301 and imposed-exit schedules ``0x400 + i``.

The workloads use an untied LM head of the embedding's shape.  A tied random
decoder reads its own input token back at the readout layer: the residual at
half depth still points along the input's embedding row, so that token's
logit dominates and every step repeats the input with probability near one.
An untied head removes that artefact; it moves the same bytes per step (the
embedding contributes one row).  ``tied_embedding=True`` remains available.
"""
from __future__ import annotations

import ctypes
import dataclasses
import math
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "libsynth.so")
_lock = threading.Lock()
_lib = None

SID_EMBED = 0x100
SID_LM_HEAD = 0x101
SID_PROMPT = 0x300
SID_CALIB = 0x301
SID_SCHEDULE = 0x400
KINDS = {"wq": 0, "wk": 1, "wv": 2, "wo": 3, "wg": 4, "wu": 5, "wd": 6, "bq": 7, "bk": 8, "bv": 9}
WEIGHT_STD = 0.02


def build(force: bool = False) -> str:
    """Compile ``libsynth.so`` with gcc (OpenMP)."""
    os.makedirs(_BUILD, exist_ok=True)
    src = os.path.join(_HERE, "synth.c")
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(src):
        tmp = _SO + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared",
                               "-o", tmp, src, "-lm"])
        os.replace(tmp, _SO)
    return _SO


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_SO)
            u64, i64, dbl = ctypes.c_uint64, ctypes.c_int64, ctypes.c_double
            vp = ctypes.c_void_p
            lib.synth_u64.argtypes = [u64, u64, u64, i64, vp]
            lib.synth_normal_bf16.argtypes = [u64, u64, i64, dbl, dbl, vp]
            lib.synth_identity_plus_normal_bf16.argtypes = [u64, u64, i64, i64, dbl, vp]
            lib.synth_fill_bf16.argtypes = [i64, dbl, vp]
            lib.synth_token_ids.argtypes = [u64, u64, i64, ctypes.c_int32, vp]
            lib.synth_bernoulli.argtypes = [u64, u64, i64, dbl, vp]
            for f in (lib.synth_u64, lib.synth_normal_bf16, lib.synth_identity_plus_normal_bf16,
                      lib.synth_fill_bf16, lib.synth_token_ids, lib.synth_bernoulli):
                f.restype = None
            _lib = lib
    return _lib


def u64_stream(seed: int, sid: int, first: int, n: int) -> np.ndarray:
    out = np.empty(n, dtype=np.uint64)
    _load().synth_u64(seed, sid, first, n, out.ctypes.data)
    return out


def normal_bf16(seed: int, sid: int, shape, std: float = WEIGHT_STD, mean: float = 0.0) -> np.ndarray:
    shape = tuple(int(s) for s in np.atleast_1d(shape))
    out = np.empty(shape, dtype=np.uint16)
    _load().synth_normal_bf16(seed, sid, out.size, mean, std, out.ctypes.data)
    return out


def identity_plus_normal_bf16(seed: int, sid: int, n: int, std: float = WEIGHT_STD) -> np.ndarray:
    out = np.empty((n, n), dtype=np.uint16)
    _load().synth_identity_plus_normal_bf16(seed, sid, n, n, std, out.ctypes.data)
    return out


def const_bf16(shape, value: float) -> np.ndarray:
    shape = tuple(int(s) for s in np.atleast_1d(shape))
    out = np.empty(shape, dtype=np.uint16)
    _load().synth_fill_bf16(out.size, value, out.ctypes.data)
    return out


def token_ids(seed: int, sid: int, n: int, vocab: int) -> np.ndarray:
    out = np.empty(n, dtype=np.int32)
    _load().synth_token_ids(seed, sid, n, vocab, out.ctypes.data)
    return out


def bernoulli(seed: int, sid: int, n: int, rate: float) -> np.ndarray:
    out = np.empty(n, dtype=np.int8)
    _load().synth_bernoulli(seed, sid, n, rate, out.ctypes.data)
    return out


def bf16_to_f32(a: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32."""
    return (np.asarray(a, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


@dataclasses.dataclass
class ModelShape:
    """Decoder shape: L layers, width d, A query / K key-value heads of size D,
    SwiGLU width F, vocabulary V."""
    name: str
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    ffn_dim: int
    vocab: int
    readout_layers: tuple
    seed: int
    prompt_len: int
    new_tokens: int
    exit_rates: tuple = ()
    rms_eps: float = 1e-6
    rope_base: float = 10000.0
    qkv_bias: bool = False
    tied_embedding: bool = False
    logit_scale: float | None = None   # s; None -> 1.5 * sqrt(2 ln V)

    @property
    def final_gain(self) -> float:
        s = self.logit_scale if self.logit_scale is not None else 1.5 * math.sqrt(2.0 * math.log(self.vocab))
        return s / (WEIGHT_STD * math.sqrt(self.d_model))

    @property
    def max_ctx(self) -> int:
        return self.prompt_len + self.new_tokens

    def replace(self, **kw) -> "ModelShape":
        return dataclasses.replace(self, **kw)


# The five workloads: shapes of Qwen2.5-0.5B / 1.5B and a 3B-like decoder,
# readouts at half depth (three readouts at 1/4, 1/2, 3/4 for the long case).
CONFIGS = {
    "tiny": ModelShape("tiny", 4, 256, 4, 2, 64, 688, 4096, (2,), 0, 32, 64, (0.0, 0.5, 1.0)),
    "0.5b": ModelShape("0.5b", 24, 896, 14, 2, 64, 4864, 151936, (12,), 1, 256, 256, (0.0, 0.5, 1.0)),
    "1.5b": ModelShape("1.5b", 28, 1536, 12, 2, 128, 8960, 151936, (14,), 2, 512, 512,
                       (0.0, 0.08, 0.5, 0.96, 1.0)),
    "3b": ModelShape("3b", 36, 2048, 16, 2, 128, 11008, 151936, (18,), 3, 1024, 512, (0.0, 0.5, 0.96)),
    "1.5b-long": ModelShape("1.5b-long", 28, 1536, 12, 2, 128, 8960, 151936, (7, 14, 21), 4, 8192, 1024,
                            (0.5,)),
}


def layer_sid(j: int, kind: str) -> int:
    return 0x1000 + 16 * j + KINDS[kind]


def make_layer(shape: ModelShape, j: int) -> dict:
    """bf16 weights of layer j (0-based)."""
    s, d = shape.seed, shape.d_model
    qd, kd, F = shape.n_heads * shape.head_dim, shape.n_kv_heads * shape.head_dim, shape.ffn_dim
    lw = {
        "attn_norm": const_bf16(d, 1.0),
        "wq": normal_bf16(s, layer_sid(j, "wq"), (qd, d)),
        "wk": normal_bf16(s, layer_sid(j, "wk"), (kd, d)),
        "wv": normal_bf16(s, layer_sid(j, "wv"), (kd, d)),
        "wo": normal_bf16(s, layer_sid(j, "wo"), (d, qd)),
        "mlp_norm": const_bf16(d, 1.0),
        "wg": normal_bf16(s, layer_sid(j, "wg"), (F, d)),
        "wu": normal_bf16(s, layer_sid(j, "wu"), (F, d)),
        "wd": normal_bf16(s, layer_sid(j, "wd"), (d, F)),
    }
    if shape.qkv_bias:
        lw["bq"] = normal_bf16(s, layer_sid(j, "bq"), qd)
        lw["bk"] = normal_bf16(s, layer_sid(j, "bk"), kd)
        lw["bv"] = normal_bf16(s, layer_sid(j, "bv"), kd)
    return lw


def make_readout(shape: ModelShape, r: int) -> tuple:
    """(layer, W_r [d, d], b_r [d]) of readout r."""
    d = shape.d_model
    w = identity_plus_normal_bf16(shape.seed, 0x200 + 2 * r, d)
    b = normal_bf16(shape.seed, 0x201 + 2 * r, d)
    return shape.readout_layers[r], w, b


def make_model(shape: ModelShape) -> dict:
    """All weights of a synthetic model plus its readouts."""
    V, d = shape.vocab, shape.d_model
    model = {
        "embed": normal_bf16(shape.seed, SID_EMBED, (V, d)),
        "lm_head": None if shape.tied_embedding else normal_bf16(shape.seed, SID_LM_HEAD, (V, d)),
        "final_norm": const_bf16(d, shape.final_gain),
        "layers": [make_layer(shape, j) for j in range(shape.n_layers)],
        "readouts": [make_readout(shape, r) for r in range(len(shape.readout_layers))],
    }
    return model


def prompt(shape: ModelShape, n: int | None = None) -> np.ndarray:
    return token_ids(shape.seed, SID_PROMPT, shape.prompt_len if n is None else n, shape.vocab)


def calibration_stream(shape: ModelShape, n: int = 2048) -> np.ndarray:
    return token_ids(shape.seed, SID_CALIB, n, shape.vocab)


def exit_schedule(shape: ModelShape, n: int, rate: float, index: int = 0) -> np.ndarray:
    """Seeded Bernoulli(rate) imposed-exit schedule (1 = exit)."""
    return bernoulli(shape.seed, SID_SCHEDULE + index, n, rate)
