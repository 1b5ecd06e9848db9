"""Section 11's full-depth re-pass on the GPU (needs a GB300).

Positions that exited keep their exit residual; ee_repass runs their skipped
layers again in position order.  Checked against the oracle's re-pass
(entries within 1e-2 relative, kv_src bit for bit), against the GPU's own
full-depth run of the same tokens (bit for bit once every exited position
has been re-passed, when the re-pass runs one position at a time), and
through the periodic option of ee_decode_n."""
import numpy as np
import pytest

import oracle
import synth
from helpers import rel_err

pytestmark = pytest.mark.gpu

TINY = synth.CONFIGS["tiny"]


@pytest.fixture(scope="module")
def tiny_model():
    return synth.make_model(TINY)


def _force(i, every=3):
    return oracle.FORCE_FULL if i % every == 0 else oracle.FORCE_EXIT_AT(0)


def _decode_both(model, n, persistent=True, graphs=True, rows=True):
    from paper_2609_14144_gb300 import OPT_GRAPHS, OPT_PERSISTENT, OPT_ROWS, Engine

    P = TINY.prompt_len
    orc = oracle.Oracle(TINY, model, max_ctx=P + n + 2)
    eng = Engine(TINY, model, max_ctx=P + n + 2)
    eng.set_option(OPT_PERSISTENT, int(persistent))
    eng.set_option(OPT_GRAPHS, int(graphs))
    eng.set_option(OPT_ROWS, int(rows))
    tok = orc.prefill(synth.prompt(TINY))
    eng.prefill(synth.prompt(TINY))
    ins = []
    for i in range(n):
        ins.append(tok)
        o = orc.decode_step(tok, [2.0], _force(i))
        eng.decode_step(tok, [2.0], _force(i))
        tok = o["token"]
    return orc, eng, ins


def _check_cache(orc, eng, t_end, tol=1e-2):
    for j in range(TINY.n_layers):
        for t in range(t_end):
            ko, vo, so = orc.kv(j, t)
            kg, vg = eng.kv(j, t)
            assert eng.kv_src(j, t) == so, (j, t)
            assert rel_err(kg, ko) <= tol and rel_err(vg, vo) <= tol, (j, t)


@pytest.mark.parametrize("persistent,rows", [(True, True), (True, False), (False, False)])
def test_tiny_repass_matches_oracle(tiny_model, persistent, rows):
    n = 18
    P = TINY.prompt_len
    orc, eng, _ = _decode_both(tiny_model, n, persistent=persistent, rows=rows)
    _check_cache(orc, eng, P + n)  # before: filled entries agree
    t0, t1 = P + 4, P + n
    assert eng.repass(t0, t1) == orc.repass(t0, t1) == sum(1 for i in range(4, n) if i % 3)
    _check_cache(orc, eng, P + n)
    assert eng.repass(t0, t1) == 0  # nothing left in the range
    assert eng.position == orc.pos == P + n
    # decoding goes on from the same position and token
    o = orc.decode_step(7, [2.0], oracle.FORCE_FULL)
    g = eng.decode_step(7, [2.0], oracle.FORCE_FULL)
    assert abs(g["confidence"][0] - o["confidence"][0]) <= 1e-3


def test_repass_gives_the_full_depth_cache_bit_for_bit(tiny_model):
    """Exits then a re-pass of every exited position, one position at a time
    through the decode step's layer kernels, equal bit for bit the GPU's own
    full-depth run of the same tokens."""
    from paper_2609_14144_gb300 import FORCE_FULL, OPT_ROWS, Engine

    n = 15
    P = TINY.prompt_len
    _, eng, ins = _decode_both(tiny_model, n, rows=False)
    assert eng.repass(P, P + n) == sum(1 for i in range(n) if i % 3)
    full = Engine(TINY, tiny_model, max_ctx=P + n + 2)
    full.set_option(OPT_ROWS, 0)
    full.prefill(synth.prompt(TINY))
    for tok in ins:
        full.decode_step(tok, [2.0], FORCE_FULL)
    for j in range(TINY.n_layers):
        for t in range(P + n):
            ka, va = eng.kv(j, t)
            kb, vb = full.kv(j, t)
            assert eng.kv_src(j, t) == full.kv_src(j, t) == 1, (j, t)
            assert np.array_equal(ka, kb) and np.array_equal(va, vb), (j, t)


def test_periodic_repass_option(tiny_model):
    """EE_OPT_REPASS = P: ee_decode_n re-passes each run of P decoded
    positions; the cache equals an explicit re-pass after the same decode."""
    from paper_2609_14144_gb300 import OPT_REPASS, Engine

    n, period = 24, 8
    P = TINY.prompt_len
    sched = np.array([0 if i % 3 == 0 else 2 for i in range(n)], np.int8)  # FORCE_FULL / FORCE_EXIT_AT(0)
    a = Engine(TINY, tiny_model, max_ctx=P + n + 2)
    a.prefill(synth.prompt(TINY))
    a.set_option(OPT_REPASS, period)
    ta, ea, _ = a.decode_n(n, [2.0], schedule=sched)
    b = Engine(TINY, tiny_model, max_ctx=P + n + 2)
    b.prefill(synth.prompt(TINY))
    tb, eb, _ = b.decode_n(n, [2.0], schedule=sched)
    assert list(ea) == list(eb)
    # the tokens of each period are decoded before its re-pass, so up to the
    # first re-pass they agree; b catches up with an explicit re-pass
    assert list(ta[:period]) == list(tb[:period])
    k = TINY.readout_layers[0]
    for t in range(P, P + n):
        assert a.kv_src(k, t) == 1, t  # every exited position was re-passed
    assert b.kv_src(k, P + 1) == 2
    assert a.position == b.position == P + n


def test_repass_api_errors(tiny_model):
    from paper_2609_14144_gb300 import EEError, Engine

    eng = Engine(TINY, tiny_model, max_ctx=TINY.prompt_len + 8)
    with pytest.raises(EEError):
        eng.repass(0, 0)  # before prefill
    eng.prefill(synth.prompt(TINY))
    for bad in ((-1, 2), (5, 3), (0, TINY.prompt_len + 1)):
        with pytest.raises(EEError):
            eng.repass(*bad)
    assert eng.repass(0, TINY.prompt_len) == 0  # prefill positions never exit


def test_1p5b_repass_sampled():
    """The 1.5B shape: a re-pass of a few exited positions against the
    oracle's, on sampled layers."""
    from paper_2609_14144_gb300 import Engine

    shape = synth.CONFIGS["1.5b"].replace(prompt_len=64)
    model = synth.make_model(shape)
    n, P = 6, 64
    orc = oracle.Oracle(shape, model, max_ctx=P + n)
    eng = Engine(shape, model, max_ctx=P + n)
    tok = orc.prefill(synth.prompt(shape))
    eng.prefill(synth.prompt(shape))
    for i in range(n):
        o = orc.decode_step(tok, [2.0], _force(i))
        eng.decode_step(tok, [2.0], _force(i))
        tok = o["token"]
    assert eng.repass(P, P + n) == orc.repass(P, P + n) == 4
    for j in (14, 20, 27):
        for t in range(P, P + n):
            ko, vo, so = orc.kv(j, t)
            kg, vg = eng.kv(j, t)
            assert eng.kv_src(j, t) == so == 1
            assert rel_err(kg, ko) <= 1e-2 and rel_err(vg, vo) <= 1e-2, (j, t)
