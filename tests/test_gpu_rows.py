"""The multi-position layer pass on the GPU (needs a GB300).

With EE_OPT_ROWS = 1 the prompt and the re-pass run each layer over batches
of up to 256 positions, the projections on the tcgen05 tensor cores (2: the
same batches with warp-level mma products).  Checked against the oracle (first token exact outside
the 1e-3 top-2 band, final hidden state and logits and every cache entry
within 1e-2 relative, which (layer, position) entries were computed bit for
bit) and against the same engine one position at a time (EE_OPT_ROWS = 0,
the default): both keep activations at fp32 precision (the batched products
through three bf16 parts of each activation), so fp32 results agree within
1e-3 relative; cache entries are bf16, where one rounding step is 4e-3."""
import numpy as np
import pytest

import oracle
import synth
from helpers import EXCLUDE_EPS, REL_TOL, check_kv, rel_err

pytestmark = pytest.mark.gpu

TINY = synth.CONFIGS["tiny"]
PATH_TOL = 1e-3  # fp32 results of the batched and the one-position paths


@pytest.fixture(scope="module")
def tiny_model():
    return synth.make_model(TINY)


def _top2_gap(logits) -> float:
    z = np.asarray(logits, np.float64)
    p = np.exp(z - z.max())
    p /= p.sum()
    a = np.sort(p)
    return float(a[-1] - a[-2])


def _engine(shape, model, max_ctx, rows=True, pages=None):
    from paper_2609_14144_gb300 import OPT_DEBUG_LOGITS, OPT_ROWS, Engine

    eng = Engine(shape, model, max_ctx=max_ctx)
    eng.set_option(OPT_ROWS, int(rows))
    eng.set_option(OPT_DEBUG_LOGITS, 1)
    if pages is not None:
        eng.set_page_table(pages)
    return eng


@pytest.mark.parametrize("mode", [1, 2])
@pytest.mark.parametrize("n", [1, 7, 16, 17, 255, 256, 257, 600])
def test_tiny_prompt_batches_match_oracle(tiny_model, n, mode):
    """Prompts of one position, a partial first group of 16 rows (the
    tcgen05 products' N step), one full group, a full group and one row, one
    short of a full batch, one full batch, a full batch and one position, and
    two full batches and a ragged tail, on the tcgen05 and the warp-level
    products (F = 688: a ragged last K stage)."""
    prompt = synth.token_ids(TINY.seed, 901, n, TINY.vocab)
    orc = oracle.Oracle(TINY, tiny_model, max_ctx=n + 1)
    tok_o, cap = orc.prefill(prompt, capture=True)
    eng = _engine(TINY, tiny_model, n + 1, rows=mode)
    tok_g = eng.prefill(prompt)
    if _top2_gap(cap["final_logits"]) >= EXCLUDE_EPS:
        assert tok_g == tok_o
    assert eng.position == n
    assert rel_err(eng.hidden_final(), cap["h_final"]) <= REL_TOL
    assert rel_err(eng.final_logits(), cap["final_logits"]) <= REL_TOL
    check_kv(orc, eng, TINY, n)


def test_tiny_prompt_permuted_pages_and_bias():
    shape = TINY.replace(qkv_bias=True)
    model = synth.make_model(shape)
    n = 260
    pages = np.random.default_rng(3).permutation((n + 1 + 63) // 64).astype(np.int32)
    prompt = synth.token_ids(shape.seed, 902, n, shape.vocab)
    orc = oracle.Oracle(shape, model, max_ctx=n + 1)
    tok_o, cap = orc.prefill(prompt, capture=True)
    eng = _engine(shape, model, n + 1, pages=pages)
    tok_g = eng.prefill(prompt)
    if _top2_gap(cap["final_logits"]) >= EXCLUDE_EPS:
        assert tok_g == tok_o
    check_kv(orc, eng, shape, n)


def test_tiny_prompt_paths_agree(tiny_model):
    """The batched prompt and the one-position path: same first token, fp32
    states within 1e-3, and the same continuation."""
    n = 300
    prompt = synth.token_ids(TINY.seed, 903, n, TINY.vocab)
    a = _engine(TINY, tiny_model, n + 9, rows=True)
    b = _engine(TINY, tiny_model, n + 9, rows=False)
    ta, tb = a.prefill(prompt), b.prefill(prompt)
    if _top2_gap(b.final_logits()) >= EXCLUDE_EPS:
        assert ta == tb
    assert rel_err(a.hidden_final(), b.hidden_final()) <= PATH_TOL
    assert rel_err(a.final_logits(), b.final_logits()) <= PATH_TOL
    for j in range(TINY.n_layers):
        for t in range(n):
            assert a.kv_src(j, t) == b.kv_src(j, t) == 1
            ka, va = a.kv(j, t)
            kb, vb = b.kv(j, t)
            assert rel_err(ka, kb) <= REL_TOL and rel_err(va, vb) <= REL_TOL, (j, t)
    tok = tb
    for _ in range(8):  # the same inputs to both
        ra = a.decode_step(tok, [2.0], oracle.FORCE_FULL)
        rb = b.decode_step(tok, [2.0], oracle.FORCE_FULL)
        if _top2_gap(b.final_logits()) >= EXCLUDE_EPS:
            assert ra["token"] == rb["token"]
        assert abs(ra["confidence"][0] - rb["confidence"][0]) <= 5e-4
        tok = rb["token"]


def _exit_decode(shape, model, n, force_of, rows=True):
    P = shape.prompt_len
    orc = oracle.Oracle(shape, model, max_ctx=P + n + 1)
    eng = _engine(shape, model, P + n + 1, rows=rows)
    tok = orc.prefill(synth.prompt(shape))
    eng.prefill(synth.prompt(shape))
    taus = [2.0] * len(shape.readout_layers)
    for i in range(n):
        o = orc.decode_step(tok, taus, force_of(i))
        eng.decode_step(tok, taus, force_of(i))
        tok = o["token"]
    return orc, eng


def test_tiny_repass_in_several_batches(tiny_model):
    """450 decoded positions, two of three exited: 300 rows, a full batch and
    a partial one."""
    n, P = 450, TINY.prompt_len
    force = lambda i: oracle.FORCE_FULL if i % 3 == 0 else oracle.FORCE_EXIT_AT(0)
    orc, eng = _exit_decode(TINY, tiny_model, n, force)
    assert eng.repass(P, P + n) == orc.repass(P, P + n) == n - (n + 2) // 3
    check_kv(orc, eng, TINY, P + n)
    assert eng.repass(P, P + n) == 0


def test_tiny_repass_rows_starting_at_different_layers():
    """Three readouts: exits at layers 1, 2 and 3 in one batch, so rows join
    the batch at different layers."""
    shape = TINY.replace(readout_layers=(1, 2, 3))
    model = synth.make_model(shape)
    n, P = 40, shape.prompt_len
    force = lambda i: oracle.FORCE_FULL if i % 4 == 3 else oracle.FORCE_EXIT_AT(i % 4)
    orc, eng = _exit_decode(shape, model, n, force)
    assert eng.repass(P + 5, P + n) == orc.repass(P + 5, P + n)
    check_kv(orc, eng, shape, P + n)


def test_tiny_repass_paths_agree(tiny_model):
    n, P = 30, TINY.prompt_len
    force = lambda i: oracle.FORCE_FULL if i % 3 == 0 else oracle.FORCE_EXIT_AT(0)
    _, a = _exit_decode(TINY, tiny_model, n, force, rows=True)
    _, b = _exit_decode(TINY, tiny_model, n, force, rows=False)
    assert a.repass(P, P + n) == b.repass(P, P + n) == 20
    for j in range(TINY.n_layers):
        for t in range(P + n):
            assert a.kv_src(j, t) == b.kv_src(j, t) == 1
            ka, va = a.kv(j, t)
            kb, vb = b.kv(j, t)
            assert rel_err(ka, kb) <= REL_TOL and rel_err(va, vb) <= REL_TOL, (j, t)
    assert rel_err(a.hidden_final(), b.hidden_final()) <= PATH_TOL  # the last re-passed position's


def test_1p5b_prompt_batches_sampled():
    """The 1.5B shape with a 300-position prompt (a full batch and a partial
    one): first token, final state and sampled cache entries."""
    shape = synth.CONFIGS["1.5b"].replace(prompt_len=300)
    model = synth.make_model(shape)
    n = 300
    prompt = synth.prompt(shape)
    orc = oracle.Oracle(shape, model, max_ctx=n + 1)
    tok_o, cap = orc.prefill(prompt, capture=True)
    eng = _engine(shape, model, n + 1)
    tok_g = eng.prefill(prompt)
    if _top2_gap(cap["final_logits"]) >= EXCLUDE_EPS:
        assert tok_g == tok_o
    assert rel_err(eng.hidden_final(), cap["h_final"]) <= REL_TOL
    for j in (0, 13, 27):
        for t in (0, 127, 128, 255, 256, 299):
            ko, vo, so = orc.kv(j, t)
            kg, vg = eng.kv(j, t)
            assert eng.kv_src(j, t) == so == 1
            assert rel_err(kg, ko) <= REL_TOL and rel_err(vg, vo) <= REL_TOL, (j, t)


@pytest.mark.parametrize("name", ["0.5b", "1.5b"])
def test_tensor_core_paths_agree(name):
    """The tcgen05 products (EE_OPT_ROWS = 1) against the warp-level ones
    (2) on a 256-position batch and a 44-position one: same first token,
    fp32 states within 1e-3, cache entries within 1e-2 (bf16 rounding)."""
    shape = synth.CONFIGS[name].replace(prompt_len=300)
    model = synth.make_model(shape)
    prompt = synth.prompt(shape)
    a = _engine(shape, model, 301, rows=1)
    b = _engine(shape, model, 301, rows=2)
    ta, tb = a.prefill(prompt), b.prefill(prompt)
    if _top2_gap(b.final_logits()) >= EXCLUDE_EPS:
        assert ta == tb
    assert rel_err(a.hidden_final(), b.hidden_final()) <= PATH_TOL
    assert rel_err(a.final_logits(), b.final_logits()) <= PATH_TOL
    for j in (0, shape.n_layers // 2, shape.n_layers - 1):
        for t in (0, 31, 127, 255, 256, 299):
            ka, va = a.kv(j, t)
            kb, vb = b.kv(j, t)
            assert rel_err(ka, kb) <= REL_TOL and rel_err(va, vb) <= REL_TOL, (j, t)
