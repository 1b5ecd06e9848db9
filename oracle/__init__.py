"""CPU oracle of the confidence-gated early-exit decode step (test infrastructure).

Only the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  It wraps ``oracle.c`` (plain C11 +
OpenMP, double accumulation), which shares no code with the CUDA library.
See the header of ``oracle.c`` for the paper passages each part follows and
for what pins it.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None

MAX_READOUTS = 8
FORCE_FREE = 0
FORCE_FULL = 1
# Section 10 confidence signals the gate may compare with tau
CONF_PMAX, CONF_MARGIN, CONF_NEGENT = 0, 1, 2


def FORCE_EXIT_AT(r: int) -> int:
    return 2 + r


def build(force: bool = False) -> str:
    """Compile ``liboracle.so`` (gcc, OpenMP)."""
    os.makedirs(_BUILD, exist_ok=True)
    src = os.path.join(_HERE, "oracle.c")
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(src):
        tmp = _SO + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared",
                               "-o", tmp, src, "-lm"])
        os.replace(tmp, _SO)
    return _SO


class Config(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("d_model", ctypes.c_int32), ("n_heads", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32), ("ffn_dim", ctypes.c_int32),
                ("vocab", ctypes.c_int32), ("max_ctx", ctypes.c_int32), ("rms_eps", ctypes.c_double),
                ("rope_base", ctypes.c_double), ("qkv_bias", ctypes.c_int32), ("bf16_activations", ctypes.c_int32)]


_P = ctypes.c_void_p
_PP = ctypes.POINTER(ctypes.c_void_p)


class Weights(ctypes.Structure):
    _fields_ = [("embed", _P), ("lm_head", _P), ("final_norm", _P), ("attn_norm", _PP), ("wq", _PP),
                ("wk", _PP), ("wv", _PP), ("bq", _PP), ("bk", _PP), ("bv", _PP), ("wo", _PP),
                ("mlp_norm", _PP), ("wg", _PP), ("wu", _PP), ("wd", _PP)]


class Conf(ctypes.Structure):
    _fields_ = [("p1", ctypes.c_float), ("p2", ctypes.c_float), ("gap", ctypes.c_float),
                ("max_logit", ctypes.c_float), ("argmax", ctypes.c_int32), ("neg_entropy", ctypes.c_float)]


class StepResult(ctypes.Structure):
    _fields_ = [("token", ctypes.c_int32), ("exited", ctypes.c_int32), ("exit_readout", ctypes.c_int32),
                ("exit_layer", ctypes.c_int32), ("n_evaluated", ctypes.c_int32), ("full_token", ctypes.c_int32),
                ("gate_pass", ctypes.c_int32 * MAX_READOUTS), ("readout_token", ctypes.c_int32 * MAX_READOUTS),
                ("confidence", ctypes.c_float * MAX_READOUTS), ("gap", ctypes.c_float * MAX_READOUTS),
                ("full_confidence", ctypes.c_float), ("full_gap", ctypes.c_float),
                ("nucleus_member", ctypes.c_int32), ("nucleus_mass", ctypes.c_float)]

    def as_dict(self) -> dict:
        n = self.n_evaluated
        return {"token": self.token, "exited": self.exited, "exit_readout": self.exit_readout,
                "exit_layer": self.exit_layer, "n_evaluated": n, "full_token": self.full_token,
                "gate_pass": list(self.gate_pass[:n]), "readout_token": list(self.readout_token[:n]),
                "confidence": list(self.confidence[:n]), "gap": list(self.gap[:n]),
                "full_confidence": self.full_confidence, "full_gap": self.full_gap,
                "nucleus_member": self.nucleus_member, "nucleus_mass": self.nucleus_mass}


class Capture(ctypes.Structure):
    _fields_ = [("h_readout", _P), ("y_readout", _P), ("readout_logits", _P), ("h_final", _P),
                ("final_logits", _P), ("layer_trace", _P)]


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_SO)
            f32p = ctypes.POINTER(ctypes.c_float)
            lib.orc_op_bf16_round.argtypes = [_P, ctypes.c_int64, _P]
            lib.orc_op_rmsnorm.argtypes = [_P, _P, ctypes.c_int, ctypes.c_double, _P]
            lib.orc_op_matvec.argtypes = [_P, _P, ctypes.c_int64, ctypes.c_int64, _P, _P]
            lib.orc_op_rope.argtypes = [_P, ctypes.c_int, ctypes.c_int64, ctypes.c_double]
            lib.orc_op_attention.argtypes = [_P, _P, _P, ctypes.c_int, ctypes.c_int, _P]
            lib.orc_op_silu.argtypes = [ctypes.c_double]
            lib.orc_op_silu.restype = ctypes.c_double
            lib.orc_op_silu_array.argtypes = [_P, ctypes.c_int64, _P]
            lib.orc_op_confidence.argtypes = [_P, ctypes.c_int64, ctypes.POINTER(Conf)]
            lib.orc_trace_layout.argtypes = [ctypes.POINTER(Config), _P]
            lib.orc_trace_layout.restype = ctypes.c_int64
            lib.orc_create.argtypes = [ctypes.POINTER(Config), ctypes.POINTER(Weights)]
            lib.orc_create.restype = _P
            lib.orc_free.argtypes = [_P]
            lib.orc_add_readout.argtypes = [_P, ctypes.c_int, _P, _P]
            lib.orc_reset.argtypes = [_P]
            lib.orc_set_confidence.argtypes = [_P, ctypes.c_int]
            lib.orc_set_nucleus.argtypes = [_P, ctypes.c_double]
            lib.orc_op_nucleus_member.argtypes = [_P, ctypes.c_int64, ctypes.c_int32, ctypes.c_double,
                                                  ctypes.POINTER(ctypes.c_double)]
            lib.orc_select_tau.argtypes = [_P, _P, ctypes.c_int, ctypes.c_double, ctypes.POINTER(ctypes.c_float)]
            lib.orc_prefill.argtypes = [_P, _P, ctypes.c_int, ctypes.POINTER(ctypes.c_int32),
                                        ctypes.POINTER(Capture)]
            lib.orc_decode_step.argtypes = [_P, ctypes.c_int32, _P, ctypes.c_int, ctypes.POINTER(StepResult),
                                            ctypes.POINTER(Capture)]
            lib.orc_position.argtypes = [_P]
            lib.orc_truncate.argtypes = [_P, ctypes.c_int]
            lib.orc_repass.argtypes = [_P, ctypes.c_int, ctypes.c_int]
            lib.orc_set_lazy_fill.argtypes = [_P, ctypes.c_int]
            lib.orc_set_gemm.argtypes = [_P, _P]
            lib.orc_flush_fills.argtypes = [_P]
            lib.orc_kv.argtypes = [_P, ctypes.c_int, ctypes.c_int, _P, _P, ctypes.POINTER(ctypes.c_int8)]
            lib.orc_stats.argtypes = [_P, _P]
            del f32p
            _lib = lib
    return _lib


def _f32(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float32)


# ---------------------------------------------------------------- ops
def bf16_round(x) -> np.ndarray:
    x = _f32(x)
    out = np.empty_like(x)
    _load().orc_op_bf16_round(x.ctypes.data, x.size, out.ctypes.data)
    return out


def rmsnorm(h, g_bf16, eps: float) -> np.ndarray:
    h = _f32(h)
    g = np.ascontiguousarray(g_bf16, dtype=np.uint16)
    out = np.empty_like(h)
    _load().orc_op_rmsnorm(h.ctypes.data, g.ctypes.data, h.size, eps, out.ctypes.data)
    return out


def matvec(W_bf16, x, b_bf16=None) -> np.ndarray:
    W = np.ascontiguousarray(W_bf16, dtype=np.uint16)
    x = _f32(x)
    b = None if b_bf16 is None else np.ascontiguousarray(b_bf16, dtype=np.uint16)
    out = np.empty(W.shape[0], dtype=np.float32)
    _load().orc_op_matvec(W.ctypes.data, None if b is None else b.ctypes.data, W.shape[0], W.shape[1],
                          x.ctypes.data, out.ctypes.data)
    return out


def rope(x, pos: int, base: float) -> np.ndarray:
    x = _f32(x).copy()
    _load().orc_op_rope(x.ctypes.data, x.size, pos, base)
    return x


def attention(q, K, V) -> np.ndarray:
    q, K, V = _f32(q), _f32(K), _f32(V)
    T, D = K.shape
    out = np.empty(D, dtype=np.float32)
    _load().orc_op_attention(q.ctypes.data, K.ctypes.data, V.ctypes.data, T, D, out.ctypes.data)
    return out


def silu(x) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float64)
    out = np.empty_like(x)
    _load().orc_op_silu_array(x.ctypes.data, x.size, out.ctypes.data)
    return out


def confidence(logits) -> dict:
    l = _f32(logits)
    c = Conf()
    _load().orc_op_confidence(l.ctypes.data, l.size, ctypes.byref(c))
    return {"p1": c.p1, "p2": c.p2, "gap": c.gap, "max_logit": c.max_logit, "argmax": c.argmax,
            "neg_entropy": c.neg_entropy}


def nucleus_member(logits, token: int, p_nuc: float = 0.9):
    """Section 2: (member, mass) -- whether `token` lies in the nucleus of
    share p_nuc, and the probability of the tokens strictly above it."""
    l = _f32(logits)
    mass = ctypes.c_double(0.0)
    r = _load().orc_op_nucleus_member(l.ctypes.data, l.size, int(token), float(p_nuc), ctypes.byref(mass))
    return bool(r), mass.value


def select_tau(conf, member, target: float = 0.9) -> float:
    """Section 4, step four: the lowest tau at which at least `target` of the
    early answers (conf > tau) are acceptable; inf if none."""
    c = _f32(conf)
    mb = np.ascontiguousarray(member, dtype=np.int32)
    tau = ctypes.c_float(0.0)
    if _load().orc_select_tau(c.ctypes.data, mb.ctypes.data, c.size, float(target), ctypes.byref(tau)) != 0:
        raise ValueError("oracle: select_tau failed")
    return tau.value


# ---------------------------------------------------------------- model
def blas_dgemm():
    """Address of a double-precision BLAS matrix product (scipy's exported
    Fortran-convention dgemm), or None when scipy is missing."""
    try:
        from scipy.linalg import cython_blas
    except Exception:
        return None
    cap = cython_blas.__pyx_capi__["dgemm"]
    api = ctypes.pythonapi
    api.PyCapsule_GetName.restype = ctypes.c_char_p
    api.PyCapsule_GetName.argtypes = [ctypes.py_object]
    api.PyCapsule_GetPointer.restype = ctypes.c_void_p
    api.PyCapsule_GetPointer.argtypes = [ctypes.py_object, ctypes.c_char_p]
    return api.PyCapsule_GetPointer(cap, api.PyCapsule_GetName(cap))


TRACE_FIELDS = ("h_in", "u_attn", "q", "k", "v", "o", "h_mid", "u_mlp", "gate", "up", "a", "h_out")


class Oracle:
    """A model instance: weights (numpy bf16 arrays, referenced, not copied),
    readouts, KV cache and position."""

    def __init__(self, shape, model: dict, *, readouts=True, bf16_activations: bool = False,
                 max_ctx: int | None = None, gemm: bool = True):
        self.lib = _load()
        self.shape = shape
        L = shape.n_layers
        self.cfg = Config(L, shape.d_model, shape.n_heads, shape.n_kv_heads, shape.head_dim, shape.ffn_dim,
                          shape.vocab, int(max_ctx or shape.max_ctx), shape.rms_eps, shape.rope_base,
                          int(shape.qkv_bias), int(bf16_activations))
        self._keep = []

        def arr(a):
            a = np.ascontiguousarray(a, dtype=np.uint16)
            self._keep.append(a)
            return a.ctypes.data

        def parr(key):
            vals = [(arr(model["layers"][j][key]) if key in model["layers"][j] else None) for j in range(L)]
            p = (ctypes.c_void_p * L)(*vals)
            self._keep.append(p)
            return ctypes.cast(p, _PP)

        w = Weights()
        w.embed = arr(model["embed"])
        w.lm_head = arr(model["lm_head"]) if model.get("lm_head") is not None else None
        w.final_norm = arr(model["final_norm"])
        for key in ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "wg", "wu", "wd"):
            setattr(w, key, parr(key))
        for key in ("bq", "bk", "bv"):
            setattr(w, key, parr(key) if shape.qkv_bias else ctypes.cast((ctypes.c_void_p * L)(), _PP))
        self._w = w
        self.ptr = self.lib.orc_create(ctypes.byref(self.cfg), ctypes.byref(w))
        if not self.ptr:
            raise ValueError("oracle: invalid configuration")
        # long prompts: the prefill's matrix products as BLAS calls (same steps)
        self.set_gemm(gemm)
        self.n_readouts = 0
        self.readout_layers = []
        if readouts:
            for layer, W, b in model.get("readouts", []):
                self.add_readout(layer, W, b)
        self.trace_stride = self.lib.orc_trace_layout(ctypes.byref(self.cfg), None)
        off = np.zeros(12, dtype=np.int64)
        self.lib.orc_trace_layout(ctypes.byref(self.cfg), off.ctypes.data)
        self.trace_offsets = off

    def __del__(self):
        if getattr(self, "ptr", None):
            self.lib.orc_free(self.ptr)
            self.ptr = None

    def add_readout(self, layer: int, W, b) -> int:
        Wa = np.ascontiguousarray(W, dtype=np.uint16)
        ba = np.ascontiguousarray(b, dtype=np.uint16)
        self._keep += [Wa, ba]
        r = self.lib.orc_add_readout(self.ptr, int(layer), Wa.ctypes.data, ba.ctypes.data)
        if r < 0:
            raise ValueError("oracle: bad readout")
        self.n_readouts += 1
        self.readout_layers.append(int(layer))
        return r

    def reset(self):
        self.lib.orc_reset(self.ptr)

    def set_nucleus(self, p_nuc: float):
        if self.lib.orc_set_nucleus(self.ptr, float(p_nuc)) != 0:
            raise ValueError("oracle: bad nucleus share")

    def set_confidence(self, kind: int):
        """Gate signal: CONF_PMAX (default), CONF_MARGIN or CONF_NEGENT (Section 10)."""
        if self.lib.orc_set_confidence(self.ptr, int(kind)) != 0:
            raise ValueError("oracle: bad confidence kind")

    def set_lazy_fill(self, on: bool):
        """Deferred KV fill: exit steps leave their skipped entries empty and
        the first later step that runs a layer fills that layer's pending
        entries first (the same projection of the same exit residual).
        Turning it off fills every pending entry."""
        if self.lib.orc_set_lazy_fill(self.ptr, int(bool(on))) != 0:
            raise ValueError("oracle: bad lazy-fill setting")

    def set_gemm(self, on: bool):
        """Prompts of 64 positions or more take their matrix products as one
        BLAS dgemm per projection and block of positions (on, when scipy is
        present), or run position by position (off)."""
        self.lib.orc_set_gemm(self.ptr, blas_dgemm() if on else None)

    def flush_fills(self):
        """Fill every entry an exit step deferred."""
        self.lib.orc_flush_fills(self.ptr)

    @property
    def pos(self) -> int:
        return self.lib.orc_position(self.ptr)

    def truncate(self, pos: int):
        """Forget positions >= pos (cache entries, exit records, step counts):
        decoding continues from pos as if they had never been decoded."""
        if self.lib.orc_truncate(self.ptr, int(pos)) != 0:
            raise ValueError("oracle: bad truncate position")

    def repass(self, t0: int, t1: int) -> int:
        """Section 11's full-depth re-pass over positions [t0, t1): every
        position there that exited runs its skipped layers from the residual it
        exited with, replacing the filled cache entries.  Returns how many
        positions were re-passed."""
        n = self.lib.orc_repass(self.ptr, int(t0), int(t1))
        if n < 0:
            raise ValueError("bad re-pass range")
        return n

    def prefill(self, ids, capture: bool = False):
        ids = np.ascontiguousarray(ids, dtype=np.int32)
        tok = ctypes.c_int32(-1)
        cap, bufs = self._capture(capture, full=True)
        rc = self.lib.orc_prefill(self.ptr, ids.ctypes.data, ids.size, ctypes.byref(tok),
                                  ctypes.byref(cap) if cap else None)
        if rc:
            raise ValueError(f"oracle prefill failed ({rc})")
        return (tok.value, bufs) if capture else tok.value

    def _capture(self, on: bool, full: bool = False, trace: bool = False):
        if not on:
            return None, None
        d, V, R, L = self.shape.d_model, self.shape.vocab, max(self.n_readouts, 1), self.shape.n_layers
        bufs = {"h_readout": np.zeros((R, d), np.float32), "y_readout": np.zeros((R, d), np.float32),
                "readout_logits": np.zeros((R, V), np.float32), "h_final": np.zeros(d, np.float32),
                "final_logits": np.zeros(V, np.float32)}
        if trace:
            bufs["layer_trace"] = np.zeros((L, self.trace_stride), np.float32)
        cap = Capture(*[bufs[k].ctypes.data if k in bufs else None for k in
                        ("h_readout", "y_readout", "readout_logits", "h_final", "final_logits", "layer_trace")])
        return cap, bufs

    def decode_step(self, in_tok: int, taus, force: int = FORCE_FREE, capture: bool = False, trace: bool = False):
        t = np.zeros(MAX_READOUTS, dtype=np.float32)
        taus = np.atleast_1d(np.asarray(taus, dtype=np.float32))
        t[: taus.size] = taus
        res = StepResult()
        cap, bufs = self._capture(capture or trace, trace=trace)
        rc = self.lib.orc_decode_step(self.ptr, int(in_tok), t.ctypes.data, int(force), ctypes.byref(res),
                                      ctypes.byref(cap) if cap else None)
        if rc:
            raise ValueError(f"oracle decode_step failed ({rc})")
        out = res.as_dict()
        if bufs is not None:
            out["capture"] = bufs
        return out

    def trace_field(self, trace: np.ndarray, layer: int, name: str) -> np.ndarray:
        i = TRACE_FIELDS.index(name)
        end = self.trace_offsets[i + 1] if i + 1 < 12 else self.trace_stride
        return trace[layer, self.trace_offsets[i]:end]

    def kv(self, layer: int, pos: int):
        n = self.shape.n_kv_heads * self.shape.head_dim
        k = np.zeros(n, np.float32)
        v = np.zeros(n, np.float32)
        src = ctypes.c_int8(0)
        if self.lib.orc_kv(self.ptr, layer, pos, k.ctypes.data, v.ctypes.data, ctypes.byref(src)):
            raise ValueError("oracle: bad kv index")
        return k, v, int(src.value)

    def stats(self) -> dict:
        out = np.zeros(2 + MAX_READOUTS, dtype=np.int64)
        self.lib.orc_stats(self.ptr, out.ctypes.data)
        return {"steps": int(out[0]), "full_steps": int(out[1]), "exits": [int(x) for x in out[2:2 + self.n_readouts]]}

    def generate(self, prompt, n_new: int, taus, force_schedule=None, capture: bool = False):
        """Prefill the prompt, then run n_new gated steps feeding each emitted
        token back.  Returns (first_token, [step results])."""
        first = self.prefill(prompt)
        tok = first
        out = []
        for i in range(n_new):
            force = FORCE_FREE if force_schedule is None else int(force_schedule[i])
            r = self.decode_step(tok, taus, force, capture=capture)
            r["input"] = tok
            out.append(r)
            tok = r["token"]
        return first, out
