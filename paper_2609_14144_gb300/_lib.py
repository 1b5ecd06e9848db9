"""ctypes declarations of the C ABI in include/ee.h (argument marshalling only)."""
from __future__ import annotations

import ctypes
import os

from . import build as _build

MAX_READOUTS = 8
EE_OK, EE_EINVAL, EE_ENOMEM, EE_ECUDA, EE_ERANGE, EE_EDEVICE, EE_ESTATE = 0, -1, -2, -3, -4, -5, -6
FREE, FORCE_FULL = 0, 1
HOST, DEVICE = 0, 1
OPT_GRAPHS, OPT_PDL, OPT_DEBUG_LOGITS, OPT_PERSISTENT, OPT_CONFIDENCE, OPT_NUCLEUS, OPT_REPASS = 1, 2, 3, 4, 5, 6, 7
OPT_ROWS = 8
OPT_WAIT_LIMIT = 9
OPT_LAZY_FILL = 11
CONF_PMAX, CONF_MARGIN, CONF_NEGENT = 0, 1, 2
DBG_HIDDEN_READOUT, DBG_READOUT_Y, DBG_HIDDEN_FINAL, DBG_READOUT_LOGITS, DBG_FINAL_LOGITS, DBG_KV, DBG_KV_SRC = \
    1, 2, 3, 4, 5, 6, 7

# Every symbol include/ee.h declares.
SYMBOLS = ("ee_workspace_bytes", "ee_create", "ee_destroy", "ee_last_error", "ee_load_weights", "ee_add_readout",
           "ee_set_page_table", "ee_reset", "ee_prefill", "ee_decode_step", "ee_decode_n", "ee_sync",
           "ee_get_stats", "ee_position", "ee_set_option", "ee_debug_read", "ee_attention_scratch_bytes",
           "ee_attention_decode", "ee_vocab_scratch_bytes", "ee_vocab_confidence", "ee_vocab_signals", "ee_profile_kernels",
           "ee_attention_decode_static", "ee_calibrate", "ee_select_tau", "ee_repass", "ee_flush_fills")
KERNELS = ("qkv", "attention", "oproj", "gateup", "down", "readout", "vocab", "kvfill", "layers")


def FORCE_EXIT_AT(r: int) -> int:
    return 2 + r


class ModelConfig(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("d_model", ctypes.c_int32), ("n_heads", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32), ("ffn_dim", ctypes.c_int32),
                ("vocab", ctypes.c_int32), ("rms_eps", ctypes.c_float), ("rope_base", ctypes.c_float),
                ("tied_embedding", ctypes.c_int32), ("qkv_bias", ctypes.c_int32), ("max_ctx", ctypes.c_int32),
                ("page_size", ctypes.c_int32), ("max_readouts", ctypes.c_int32)]


_P = ctypes.c_void_p
_PP = ctypes.POINTER(ctypes.c_void_p)


class HostWeights(ctypes.Structure):
    _fields_ = [("embed", _P), ("lm_head", _P), ("final_norm", _P), ("attn_norm", _PP), ("wq", _PP), ("wk", _PP),
                ("wv", _PP), ("bq", _PP), ("bk", _PP), ("bv", _PP), ("wo", _PP), ("mlp_norm", _PP), ("wg", _PP),
                ("wu", _PP), ("wd", _PP)]


class StepResult(ctypes.Structure):
    _fields_ = [("token", ctypes.c_int32), ("exited", ctypes.c_int32), ("exit_readout", ctypes.c_int32),
                ("exit_layer", ctypes.c_int32), ("n_evaluated", ctypes.c_int32), ("full_token", ctypes.c_int32),
                ("gate_pass", ctypes.c_int32 * MAX_READOUTS), ("readout_token", ctypes.c_int32 * MAX_READOUTS),
                ("confidence", ctypes.c_float * MAX_READOUTS), ("full_confidence", ctypes.c_float),
                ("nucleus_member", ctypes.c_int32), ("nucleus_mass", ctypes.c_float)]

    def as_dict(self) -> dict:
        n = self.n_evaluated
        return {"token": self.token, "exited": self.exited, "exit_readout": self.exit_readout,
                "exit_layer": self.exit_layer, "n_evaluated": n, "full_token": self.full_token,
                "gate_pass": list(self.gate_pass[:n]), "readout_token": list(self.readout_token[:n]),
                "confidence": list(self.confidence[:n]), "full_confidence": self.full_confidence,
                "nucleus_member": self.nucleus_member, "nucleus_mass": self.nucleus_mass}


class Stats(ctypes.Structure):
    _fields_ = [("steps", ctypes.c_int64), ("full_steps", ctypes.c_int64),
                ("exits", ctypes.c_int64 * MAX_READOUTS)]


_lib = None


def lib_path() -> str:
    return _build.LIB


def load(allow_build: bool = False):
    """Load libee.so; raise if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    path = lib_path()
    if not os.path.exists(path):
        if not allow_build:
            raise RuntimeError(f"{path} is missing: run __graft_entry__.build() (or "
                               "python paper_2609_14144_gb300/build.py) first")
        _build.build()
    lib = ctypes.CDLL(path)
    i32, sz = ctypes.c_int32, ctypes.c_size_t
    cfgp = ctypes.POINTER(ModelConfig)
    lib.ee_workspace_bytes.argtypes = [cfgp, ctypes.POINTER(sz)]
    lib.ee_create.argtypes = [cfgp, _P, sz, _P, ctypes.POINTER(_P)]
    lib.ee_destroy.argtypes = [_P]
    lib.ee_last_error.argtypes = []
    lib.ee_last_error.restype = ctypes.c_char_p
    lib.ee_load_weights.argtypes = [_P, ctypes.POINTER(HostWeights)]
    lib.ee_add_readout.argtypes = [_P, ctypes.c_int, _P, _P, ctypes.POINTER(ctypes.c_int)]
    lib.ee_set_page_table.argtypes = [_P, _P, ctypes.c_int]
    lib.ee_reset.argtypes = [_P]
    lib.ee_prefill.argtypes = [_P, _P, ctypes.c_int, ctypes.POINTER(i32)]
    lib.ee_decode_step.argtypes = [_P, i32, _P, ctypes.c_int, ctypes.POINTER(StepResult)]
    lib.ee_decode_n.argtypes = [_P, ctypes.c_int, i32, _P, _P, _P, _P, _P, ctypes.c_int]
    lib.ee_sync.argtypes = [_P]
    lib.ee_flush_fills.argtypes = [_P]
    lib.ee_get_stats.argtypes = [_P, ctypes.POINTER(Stats)]
    lib.ee_position.argtypes = [_P, ctypes.POINTER(i32)]
    lib.ee_set_option.argtypes = [_P, ctypes.c_int, ctypes.c_int]
    lib.ee_debug_read.argtypes = [_P, ctypes.c_int, ctypes.c_int, ctypes.c_int, _P, sz]
    lib.ee_attention_scratch_bytes.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.POINTER(sz)]
    lib.ee_attention_decode.argtypes = [_P, _P, _P, _P, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                        ctypes.c_int, _P, sz, _P, _P]
    lib.ee_vocab_scratch_bytes.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.POINTER(sz)]
    lib.ee_vocab_confidence.argtypes = [_P, _P, _P, ctypes.c_int, ctypes.c_int, ctypes.c_float, _P, sz, _P, _P, _P,
                                        _P]
    lib.ee_vocab_signals.argtypes = [_P, _P, _P, ctypes.c_int, ctypes.c_int, ctypes.c_float, _P, sz, _P, _P, _P, _P]
    lib.ee_profile_kernels.argtypes = [_P, ctypes.c_int, _P]
    lib.ee_attention_decode_static.argtypes = [_P, _P, _P, _P, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                               ctypes.c_int, _P, _P]
    lib.ee_repass.argtypes = [_P, i32, i32, ctypes.POINTER(i32)]
    lib.ee_calibrate.argtypes = [_P, _P, ctypes.c_int, ctypes.c_float, _P, _P, _P, ctypes.c_int]
    lib.ee_select_tau.argtypes = [_P, ctypes.c_int, _P, ctypes.c_int, ctypes.c_float, _P, _P, _P]
    for name in SYMBOLS:
        f = getattr(lib, name)
        if name != "ee_last_error":
            f.restype = ctypes.c_int
    _lib = lib
    return lib


class EEError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"libee error {code}: {msg}")
        self.code = code


def check(rc: int):
    if rc != EE_OK:
        msg = _lib.ee_last_error().decode() if _lib is not None else ""
        raise EEError(rc, msg)
