"""The C-ABI library builds, loads and exports every entry point that
include/ee.h declares; host-only calls validate their arguments (no GPU)."""
import ctypes
import os
import re

import pytest

import synth
from paper_2609_14144_gb300 import _lib

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    src = open(os.path.join(ROOT, "include", "ee.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:int|const char\*)\s+(ee_\w+)\s*\(", src, flags=re.M)))


@pytest.fixture(scope="module")
def lib():
    return _lib.load(allow_build=True)


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert len(names) >= 20
    assert set(names) == set(_lib.SYMBOLS)
    for n in names:
        assert hasattr(lib, n), n


def _cfg(shape, **kw):
    c = _lib.ModelConfig(shape.n_layers, shape.d_model, shape.n_heads, shape.n_kv_heads, shape.head_dim,
                         shape.ffn_dim, shape.vocab, shape.rms_eps, shape.rope_base, 0, 0, shape.max_ctx, 64, 1)
    for k, v in kw.items():
        setattr(c, k, v)
    return c


def test_workspace_bytes_and_validation(lib):
    sz = ctypes.c_size_t(0)
    sh = synth.CONFIGS["1.5b"]
    assert lib.ee_workspace_bytes(ctypes.byref(_cfg(sh)), ctypes.byref(sz)) == 0
    # weights (untied: embedding and LM head) dominate: about 3.5 GB at 1.5B
    assert 3.3e9 < sz.value < 4.0e9
    tied = ctypes.c_size_t(0)
    assert lib.ee_workspace_bytes(ctypes.byref(_cfg(sh, tied_embedding=1)), ctypes.byref(tied)) == 0
    # the vocabulary pass reads a tile-packed copy of the unembedding, so a
    # tied model still stores the row-major embedding (token lookup) and the
    # packed head: the same bytes as an untied one
    assert tied.value == sz.value
    for bad in (dict(head_dim=96), dict(n_kv_heads=5), dict(page_size=48), dict(d_model=100), dict(max_readouts=9),
                dict(vocab=0), dict(n_heads=24, n_kv_heads=2)):
        assert lib.ee_workspace_bytes(ctypes.byref(_cfg(sh, **bad)), ctypes.byref(sz)) == _lib.EE_EINVAL, bad
        assert lib.ee_last_error()
    assert lib.ee_workspace_bytes(None, ctypes.byref(sz)) == _lib.EE_EINVAL


def test_scratch_sizes_and_null_contexts(lib):
    sz = ctypes.c_size_t(0)
    assert lib.ee_attention_scratch_bytes(12, 2, 128, ctypes.byref(sz)) == 0 and sz.value > 12 * 128 * 4
    assert lib.ee_attention_scratch_bytes(12, 2, 96, ctypes.byref(sz)) == _lib.EE_EINVAL
    assert lib.ee_vocab_scratch_bytes(151936, 1536, ctypes.byref(sz)) == 0 and sz.value > 0
    assert lib.ee_vocab_scratch_bytes(151936, 100, ctypes.byref(sz)) == _lib.EE_EINVAL
    for f in (lib.ee_reset, lib.ee_sync):
        assert f(None) == _lib.EE_EINVAL
    assert lib.ee_destroy(None) == 0


def test_option_constants_match_the_header():
    """Every EE_OPT_* value include/ee.h defines is the binding's OPT_* value."""
    src = open(os.path.join(ROOT, "include", "ee.h")).read()
    defs = dict(re.findall(r"^#define EE_OPT_(\w+)\s+(\d+)", src, flags=re.M))
    assert len(defs) >= 8
    for name, value in defs.items():
        assert getattr(_lib, "OPT_" + name) == int(value), name
