"""GB300-native confidence-gated early-exit decode (arxiv 2609.14144).

Thin Python binding over libee (include/ee.h).  Every step of the decode path
runs in the library's CUDA kernels; this module only marshals arguments.
PyTorch provides device memory (the workspace tensor) and the CUDA stream.
"""
from __future__ import annotations

import ctypes

import numpy as np

from . import _lib
from ._lib import (CONF_MARGIN, CONF_NEGENT, CONF_PMAX, DEVICE, FORCE_FULL, FREE, HOST, MAX_READOUTS,
                   OPT_CONFIDENCE, OPT_DEBUG_LOGITS, OPT_GRAPHS, OPT_NUCLEUS, OPT_PDL, OPT_PERSISTENT, OPT_REPASS,
                   OPT_LAZY_FILL, OPT_ROWS, OPT_WAIT_LIMIT,
                   EEError, FORCE_EXIT_AT, check)

__all__ = ["Engine", "EEError", "FREE", "FORCE_FULL", "FORCE_EXIT_AT", "HOST", "DEVICE", "attention_decode",
           "vocab_confidence", "vocab_signals", "select_tau", "library_path"]


def library_path() -> str:
    return _lib.lib_path()


def _u16(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.uint16)


class Engine:
    """One decode context on one GPU: frozen weights, readouts, paged KV cache."""

    def __init__(self, shape, model: dict, *, max_ctx: int | None = None, page_size: int = 64,
                 device: int = 0, stream=None, readouts: bool = True, max_readouts: int | None = None):
        import torch

        self.lib = _lib.load()
        self.shape = shape
        self.device = torch.device("cuda", device)
        n_ro = len(model.get("readouts", [])) if readouts else 0
        self.cfg = _lib.ModelConfig(shape.n_layers, shape.d_model, shape.n_heads, shape.n_kv_heads, shape.head_dim,
                                    shape.ffn_dim, shape.vocab, shape.rms_eps, shape.rope_base,
                                    int(model.get("lm_head") is None), int(shape.qkv_bias),
                                    int(max_ctx or shape.max_ctx), page_size,
                                    int(max_readouts if max_readouts is not None else max(n_ro, 1)))
        nbytes = ctypes.c_size_t(0)
        check(self.lib.ee_workspace_bytes(ctypes.byref(self.cfg), ctypes.byref(nbytes)))
        self.workspace_bytes = nbytes.value
        self.workspace = torch.empty(self.workspace_bytes, dtype=torch.uint8, device=self.device)
        self.stream = stream if stream is not None else torch.cuda.Stream(device=self.device)
        ctx = ctypes.c_void_p()
        with torch.cuda.device(self.device):
            check(self.lib.ee_create(ctypes.byref(self.cfg), ctypes.c_void_p(self.workspace.data_ptr()),
                                     self.workspace_bytes, ctypes.c_void_p(self.stream.cuda_stream),
                                     ctypes.byref(ctx)))
        self.ctx = ctx
        # the persistent layer kernel is on by default where the shape allows it
        self.persistent = self.lib.ee_set_option(self.ctx, OPT_PERSISTENT, 1) == 0
        self.n_readouts = 0
        self.readout_layers = []
        self.load_weights(model)
        if readouts:
            for layer, W, b in model.get("readouts", []):
                self.add_readout(layer, W, b)

    # ------------------------------------------------------------ setup
    def load_weights(self, model: dict):
        L = self.shape.n_layers
        keep = []

        def arr(a):
            a = _u16(a)
            keep.append(a)
            return a.ctypes.data

        def parr(key):
            vals = [arr(model["layers"][j][key]) if key in model["layers"][j] else None for j in range(L)]
            p = (ctypes.c_void_p * L)(*vals)
            keep.append(p)
            return ctypes.cast(p, ctypes.POINTER(ctypes.c_void_p))

        w = _lib.HostWeights()
        w.embed = arr(model["embed"])
        w.lm_head = arr(model["lm_head"]) if model.get("lm_head") is not None else None
        w.final_norm = arr(model["final_norm"])
        for key in ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "wg", "wu", "wd"):
            setattr(w, key, parr(key))
        if self.shape.qkv_bias:
            for key in ("bq", "bk", "bv"):
                setattr(w, key, parr(key))
        check(self.lib.ee_load_weights(self.ctx, ctypes.byref(w)))

    def add_readout(self, layer: int, W, b) -> int:
        Wa, ba = _u16(W), _u16(b)
        rid = ctypes.c_int(-1)
        check(self.lib.ee_add_readout(self.ctx, int(layer), Wa.ctypes.data, ba.ctypes.data, ctypes.byref(rid)))
        self.n_readouts += 1
        self.readout_layers.append(int(layer))
        return rid.value

    def set_option(self, option: int, value: int):
        check(self.lib.ee_set_option(self.ctx, option, int(value)))
        if option == OPT_PERSISTENT:
            self.persistent = bool(value)

    def set_page_table(self, pages):
        p = np.ascontiguousarray(pages, dtype=np.int32)
        check(self.lib.ee_set_page_table(self.ctx, p.ctypes.data, p.size))

    def reset(self):
        check(self.lib.ee_reset(self.ctx))

    def close(self):
        if getattr(self, "ctx", None):
            self.lib.ee_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # ------------------------------------------------------------ hot path
    def _taus(self, taus) -> np.ndarray:
        t = np.full(MAX_READOUTS, 2.0, dtype=np.float32)
        if taus is not None:
            taus = np.atleast_1d(np.asarray(taus, dtype=np.float32))
            t[: taus.size] = taus
        return t

    def prefill(self, ids) -> int:
        ids = np.ascontiguousarray(ids, dtype=np.int32)
        tok = ctypes.c_int32(-1)
        check(self.lib.ee_prefill(self.ctx, ids.ctypes.data, ids.size, ctypes.byref(tok)))
        return tok.value

    def decode_step(self, input_token: int = -1, taus=None, force: int = FREE) -> dict:
        t = self._taus(taus)
        res = _lib.StepResult()
        check(self.lib.ee_decode_step(self.ctx, int(input_token), t.ctypes.data, int(force), ctypes.byref(res)))
        return res.as_dict()

    def decode_n(self, n: int, taus=None, input_token: int = -1, schedule=None, where: int = HOST,
                 tokens=None, exit_readout=None, confidence=None):
        """n steps with on-device token feedback.  where=HOST returns numpy
        arrays; where=DEVICE writes the given torch tensors (or allocates them)
        and returns without synchronising."""
        import torch

        t = self._taus(taus)
        sched = None if schedule is None else np.ascontiguousarray(schedule, dtype=np.int8)
        sp = None if sched is None else sched.ctypes.data
        if where == HOST:
            tok = np.zeros(n, np.int32)
            ex = np.zeros(n, np.int32)
            cf = np.zeros(n, np.float32)
            check(self.lib.ee_decode_n(self.ctx, int(n), int(input_token), t.ctypes.data, sp, tok.ctypes.data,
                                       ex.ctypes.data, cf.ctypes.data, HOST))
            return tok, ex, cf
        if tokens is None:
            tokens = torch.empty(n, dtype=torch.int32, device=self.device)
        if exit_readout is None:
            exit_readout = torch.empty(n, dtype=torch.int32, device=self.device)
        if confidence is None:
            confidence = torch.empty(n, dtype=torch.float32, device=self.device)
        check(self.lib.ee_decode_n(self.ctx, int(n), int(input_token), t.ctypes.data, sp, tokens.data_ptr(),
                                   exit_readout.data_ptr(), confidence.data_ptr(), DEVICE))
        return tokens, exit_readout, confidence

    def calibrate(self, ids, p_nuc: float = 0.9, where: int = HOST, conf=None, member=None, mass=None):
        """Teacher-forced full-depth pass over ids recording every readout's
        confidence and whether readout 0's token lies in the full model's
        nucleus of share p_nuc (Section 2 acceptance, Section 4 step four).
        where=HOST: ids is a host sequence, returns numpy (conf [n, R], member
        [n], mass [n]); where=DEVICE: ids is an int32 CUDA tensor, the given
        (or new) tensors are filled without synchronising."""
        import torch

        R = self.n_readouts
        if where == HOST:
            a = np.ascontiguousarray(ids, dtype=np.int32)
            n = a.size
            cf = np.zeros((n, R), np.float32)
            mb = np.zeros(n, np.int32)
            ms = np.zeros(n, np.float32)
            check(self.lib.ee_calibrate(self.ctx, a.ctypes.data, int(n), float(p_nuc), cf.ctypes.data, mb.ctypes.data,
                                        ms.ctypes.data, HOST))
            return cf, mb, ms
        n = ids.numel()
        if conf is None:
            conf = torch.empty((n, R), dtype=torch.float32, device=self.device)
        if member is None:
            member = torch.empty(n, dtype=torch.int32, device=self.device)
        if mass is None:
            mass = torch.empty(n, dtype=torch.float32, device=self.device)
        check(self.lib.ee_calibrate(self.ctx, ids.data_ptr(), int(n), float(p_nuc), conf.data_ptr(),
                                    member.data_ptr(), mass.data_ptr(), DEVICE))
        return conf, member, mass

    def repass(self, t0: int, t1: int) -> int:
        """Section 11's full-depth re-pass over positions [t0, t1): returns the
        number of exited positions whose skipped layers were run again."""
        n = ctypes.c_int32(0)
        check(self.lib.ee_repass(self.ctx, int(t0), int(t1), ctypes.byref(n)))
        return n.value

    def flush_fills(self):
        """Fill every key/value entry the deferred fill left pending."""
        check(self.lib.ee_flush_fills(self.ctx))

    def sync(self):
        check(self.lib.ee_sync(self.ctx))

    def stats(self) -> dict:
        s = _lib.Stats()
        check(self.lib.ee_get_stats(self.ctx, ctypes.byref(s)))
        return {"steps": s.steps, "full_steps": s.full_steps, "exits": [int(x) for x in s.exits[: self.n_readouts]]}

    @property
    def position(self) -> int:
        p = ctypes.c_int32(0)
        check(self.lib.ee_position(self.ctx, ctypes.byref(p)))
        return p.value

    def profile_kernels(self, iters: int = 56) -> dict:
        """Average device ms of each decode kernel (direct launches, CUDA events)."""
        out = np.zeros(len(_lib.KERNELS), np.float32)
        check(self.lib.ee_profile_kernels(self.ctx, int(iters), out.ctypes.data))
        return {k: float(v) for k, v in zip(_lib.KERNELS, out)}

    # ------------------------------------------------------------ debug
    def _read(self, what: int, layer: int, pos: int, out: np.ndarray) -> np.ndarray:
        check(self.lib.ee_debug_read(self.ctx, what, layer, pos, out.ctypes.data, out.nbytes))
        return out

    def hidden_at_readout(self, r: int) -> np.ndarray:
        return self._read(_lib.DBG_HIDDEN_READOUT, r, 0, np.zeros(self.shape.d_model, np.float32))

    def readout_output(self, r: int) -> np.ndarray:
        return self._read(_lib.DBG_READOUT_Y, r, 0, np.zeros(self.shape.d_model, np.float32))

    def hidden_final(self) -> np.ndarray:
        return self._read(_lib.DBG_HIDDEN_FINAL, 0, 0, np.zeros(self.shape.d_model, np.float32))

    def readout_logits(self, r: int) -> np.ndarray:
        return self._read(_lib.DBG_READOUT_LOGITS, r, 0, np.zeros(self.shape.vocab, np.float32))

    def final_logits(self) -> np.ndarray:
        return self._read(_lib.DBG_FINAL_LOGITS, 0, 0, np.zeros(self.shape.vocab, np.float32))

    def kv(self, layer: int, pos: int):
        n = self.shape.n_kv_heads * self.shape.head_dim
        raw = self._read(_lib.DBG_KV, layer, pos, np.zeros(2 * n, np.uint16))
        f = (raw.astype(np.uint32) << 16).view(np.float32)
        return f[:n].copy(), f[n:].copy()

    def kv_src(self, layer: int, pos: int) -> int:
        return int(self._read(_lib.DBG_KV_SRC, layer, pos, np.zeros(1, np.int8))[0])


# ---------------------------------------------------------------- standalone kernels
def attention_decode(q, k_pages, v_pages, page_table, T: int, n_heads: int, n_kv_heads: int, head_dim: int,
                     page_size: int, out=None, scratch=None, stream=None):
    """Split-K decode attention over a paged bf16 cache (torch CUDA tensors:
    q fp32 [A*D], pages bf16/int16 [n_pages, K, page_size, D], page_table int32)."""
    import torch

    lib = _lib.load()
    nb = ctypes.c_size_t(0)
    check(lib.ee_attention_scratch_bytes(n_heads, n_kv_heads, head_dim, ctypes.byref(nb)))
    if scratch is None:
        scratch = torch.empty(nb.value, dtype=torch.uint8, device=q.device)
    if out is None:
        out = torch.empty(n_heads * head_dim, dtype=torch.float32, device=q.device)
    s = stream if stream is not None else torch.cuda.current_stream(q.device)
    check(lib.ee_attention_decode(q.data_ptr(), k_pages.data_ptr(), v_pages.data_ptr(), page_table.data_ptr(), int(T),
                                  n_heads, n_kv_heads, head_dim, page_size, scratch.data_ptr(), scratch.numel(),
                                  out.data_ptr(), s.cuda_stream))
    return out


def vocab_confidence(x, gain, U, eps: float, logits=None, scratch=None, stream=None):
    """One unembedding pass with the confidence statistics (torch CUDA tensors:
    x fp32 [d], gain bf16 [d], U bf16 [V, d]).  Returns (token, p) tensors."""
    import torch

    lib = _lib.load()
    V, d = U.shape
    nb = ctypes.c_size_t(0)
    check(lib.ee_vocab_scratch_bytes(V, d, ctypes.byref(nb)))
    if scratch is None:
        scratch = torch.empty(nb.value, dtype=torch.uint8, device=x.device)
    tok = torch.empty(1, dtype=torch.int32, device=x.device)
    p = torch.empty(1, dtype=torch.float32, device=x.device)
    s = stream if stream is not None else torch.cuda.current_stream(x.device)
    check(lib.ee_vocab_confidence(x.data_ptr(), gain.data_ptr(), U.data_ptr(), V, d, float(eps), scratch.data_ptr(),
                                  scratch.numel(), tok.data_ptr(), p.data_ptr(),
                                  None if logits is None else logits.data_ptr(), s.cuda_stream))
    return tok, p


def vocab_signals(x, gain, U, eps: float, logits=None, scratch=None, stream=None):
    """The same pass returning (token, signals): signals is a float32 tensor
    [3] = (top-1 probability, margin to the second-best, negative entropy)."""
    import torch

    lib = _lib.load()
    V, d = U.shape
    nb = ctypes.c_size_t(0)
    check(lib.ee_vocab_scratch_bytes(V, d, ctypes.byref(nb)))
    if scratch is None:
        scratch = torch.empty(nb.value, dtype=torch.uint8, device=x.device)
    tok = torch.empty(1, dtype=torch.int32, device=x.device)
    sig = torch.empty(3, dtype=torch.float32, device=x.device)
    s = stream if stream is not None else torch.cuda.current_stream(x.device)
    check(lib.ee_vocab_signals(x.data_ptr(), gain.data_ptr(), U.data_ptr(), V, d, float(eps), scratch.data_ptr(),
                               scratch.numel(), tok.data_ptr(), sig.data_ptr(),
                               None if logits is None else logits.data_ptr(), s.cuda_stream))
    return tok, sig


def select_tau(conf, member, target: float, tau=None, scratch=None, stream=None):
    """Section 4, step four on the device: the lowest tau at which at least
    `target` of the early answers (conf > tau) are acceptable (member != 0);
    -inf when every answer may exit, +inf when no threshold reaches the
    target.  conf: float32 CUDA tensor [n] or a column of [n, R] (any stride);
    member: int32 CUDA tensor [n].  Returns a float32 tensor [1]."""
    import torch

    lib = _lib.load()
    n = member.numel()
    if conf.dim() != 1 or conf.numel() != n or conf.dtype != torch.float32 or member.dtype != torch.int32:
        raise ValueError("conf must be float32 [n] and member int32 [n]")
    if not member.is_contiguous():
        raise ValueError("member must be contiguous")
    if tau is None:
        tau = torch.empty(1, dtype=torch.float32, device=conf.device)
    if scratch is None:
        scratch = torch.empty(2, dtype=torch.int32, device=conf.device)
    s = stream if stream is not None else torch.cuda.current_stream(conf.device)
    check(lib.ee_select_tau(conf.data_ptr(), int(conf.stride(0)), member.data_ptr(), int(n), float(target),
                            tau.data_ptr(), scratch.data_ptr(), s.cuda_stream))
    return tau
