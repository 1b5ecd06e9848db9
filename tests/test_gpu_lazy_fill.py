"""The deferred key/value fill (EE_OPT_LAZY_FILL) against the oracle's
(needs a GB300).

Section 4, step five supplies a skipped layer's entries from the exit-layer
state; with the fill deferred, an exit step only records that state and the
next step that runs the layer fills every pending entry first.  Both sides
defer: tokens, gate verdicts and exit counts follow the comparison rule, the
computed/empty/filled marks agree bit for bit before and after an explicit
flush, and after the flush every cache value is within 1e-2 of the oracle's.
"""
import numpy as np
import pytest

import oracle
import synth
from helpers import check_exit_counts, check_kv, check_records, gpu_replay, oracle_steps

pytestmark = pytest.mark.gpu


def _lazy_pair(shape, model, max_ctx, persistent=True):
    from paper_2609_14144_gb300 import OPT_DEBUG_LOGITS, OPT_LAZY_FILL, OPT_PERSISTENT, Engine

    orc = oracle.Oracle(shape, model, max_ctx=max_ctx)
    orc.set_lazy_fill(True)
    eng = Engine(shape, model, max_ctx=max_ctx)
    eng.set_option(OPT_PERSISTENT, 1 if persistent else 0)
    eng.set_option(OPT_LAZY_FILL, 1)
    eng.set_option(OPT_DEBUG_LOGITS, 1)
    return orc, eng


def _marks(orc, eng, shape, n_pos):
    for j in range(shape.n_layers):
        for t in range(n_pos):
            assert eng.kv_src(j, t) == orc.kv(j, t)[2], (j, t)


@pytest.mark.parametrize("persistent", [True, False])
@pytest.mark.parametrize("readouts", [(2,), (1, 2, 3)])
def test_tiny_deferred_fill_matches_oracle(persistent, readouts):
    shape = synth.CONFIGS["tiny"].replace(readout_layers=readouts)
    model = synth.make_model(shape)
    taus = [0.45] * len(readouts)
    orc, eng = _lazy_pair(shape, model, shape.max_ctx, persistent)
    prompt = synth.prompt(shape)
    first = orc.prefill(prompt)
    assert eng.prefill(prompt) == first
    recs = gpu_replay(eng, oracle_steps(orc, first, shape.new_tokens, taus), taus)
    assert check_records(recs, taus) <= shape.new_tokens // 8
    check_exit_counts(recs, taus, len(readouts))
    exits = sum(r["o"]["exited"] for r in recs)
    assert 0 < exits < len(recs)
    # pending entries are empty (0) on both sides until a step runs their layer
    _marks(orc, eng, shape, shape.max_ctx)
    orc.flush_fills()
    eng.flush_fills()
    check_kv(orc, eng, shape, shape.max_ctx)


def test_tiny_deferred_fill_then_repass():
    """A re-pass over exited positions with fills still pending: the GPU
    flushes first, the oracle fills each layer before running it; after a
    flush both caches hold the full-depth entries of the re-passed range."""
    shape = synth.CONFIGS["tiny"]
    model = synth.make_model(shape)
    orc, eng = _lazy_pair(shape, model, shape.max_ctx)
    prompt = synth.prompt(shape)
    first = orc.prefill(prompt)
    eng.prefill(prompt)
    recs = gpu_replay(eng, oracle_steps(orc, first, 24, [0.3], capture=False), [0.3], capture=False)
    check_records(recs, [0.3], capture=False)
    P = len(prompt)
    assert orc.repass(P, P + 16) == eng.repass(P, P + 16)
    orc.flush_fills()
    eng.flush_fills()
    check_kv(orc, eng, shape, P + 24)


def test_1p5b_deferred_fill_with_runs_of_exits():
    """1.5B shape at a threshold that exits about three steps in four, so a
    full step finds several positions pending at once."""
    shape = synth.CONFIGS["1.5b"].replace(prompt_len=128, new_tokens=32)
    model = synth.make_model(shape)
    orc, eng = _lazy_pair(shape, model, shape.max_ctx)
    prompt = synth.prompt(shape)
    first = orc.prefill(prompt)
    assert eng.prefill(prompt) == first
    tau = [0.3]
    recs = gpu_replay(eng, oracle_steps(orc, first, shape.new_tokens, tau), tau)
    check_records(recs, tau)
    check_exit_counts(recs, tau, 1)
    ex = [r["o"]["exited"] for r in recs]
    runs = sum(1 for a, b in zip(ex, ex[1:]) if a and b)
    assert runs > 0 and not all(ex)
    P = len(prompt)
    pairs = [(j, t) for j in (0, 13, 14, 20, 27) for t in range(P - 2, P + shape.new_tokens)]
    for j, t in pairs:
        assert eng.kv_src(j, t) == orc.kv(j, t)[2], (j, t)
    orc.flush_fills()
    eng.flush_fills()
    check_kv(orc, eng, shape, 0, pairs=pairs)
