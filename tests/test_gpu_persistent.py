"""The persistent layer-segment kernel (EE_OPT_PERSISTENT, the default) against
the CPU oracle under teacher forcing with small pages and other shapes, and
against the five-launch path (needs a GB300).  Same parity rules as
test_gpu_parity."""
import numpy as np
import pytest

import oracle
import synth
from helpers import check_kv, check_records, gpu_replay, oracle_steps, teacher_forced

pytestmark = pytest.mark.gpu

TINY = synth.CONFIGS["tiny"]


@pytest.fixture(scope="module")
def tiny_model():
    return synth.make_model(TINY)


@pytest.mark.parametrize("tau", [0.5, 0.0, 1.01])
def test_tiny_persistent_teacher_forced(tiny_model, tau):
    n = TINY.new_tokens
    fo, fg, recs, orc, eng = teacher_forced(TINY, tiny_model, n, [tau], persistent=True)
    assert fo == fg
    excluded = check_records(recs, [tau])
    assert excluded <= n // 8
    check_kv(orc, eng, TINY, TINY.prompt_len + n)
    assert eng.stats()["exits"] == orc.stats()["exits"]


def test_tiny_persistent_permuted_small_pages(tiny_model):
    n = TINY.new_tokens
    pages = (TINY.max_ctx + 15) // 16
    perm = np.random.default_rng(1).permutation(pages).astype(np.int32)
    fo, fg, recs, orc, eng = teacher_forced(TINY, tiny_model, n, [0.5], page_perm=perm, page_size=16,
                                            persistent=True)
    assert fo == fg
    check_records(recs, [0.5])
    check_kv(orc, eng, TINY, TINY.max_ctx)


def test_tiny_persistent_eager_matches_graphs(tiny_model):
    _, _, a, _, _ = teacher_forced(TINY, tiny_model, 24, [0.5], capture=False, persistent=True)
    _, _, b, _, _ = teacher_forced(TINY, tiny_model, 24, [0.5], capture=False, graphs=False, persistent=True)
    for x, y in zip(a, b):
        assert x["g"] == y["g"]


def test_half_b_persistent_teacher_forced():
    """0.5B: d 896 (a ragged last 256-column chunk), 14/2 heads of 64."""
    shape = synth.CONFIGS["0.5b"].replace(prompt_len=48, new_tokens=12)
    model = synth.make_model(shape)
    fo, fg, recs, orc, eng = teacher_forced(shape, model, shape.new_tokens, [0.5], persistent=True)
    assert fo == fg
    check_records(recs, [0.5])
    check_kv(orc, eng, shape, shape.max_ctx)


def test_1p5b_persistent_teacher_forced():
    shape = synth.CONFIGS["1.5b"].replace(new_tokens=6)
    model = synth.make_model(shape)
    fo, fg, recs, orc, eng = teacher_forced(shape, model, shape.new_tokens, [0.5], persistent=True)
    assert fo == fg
    check_records(recs, [0.5])
    for j in (0, 13, 14, 27):
        for t in (0, 511, 512, shape.max_ctx - 1):
            assert eng.kv_src(j, t) == orc.kv(j, t)[2]


def test_1p5b_long_persistent_three_readouts():
    shape = synth.CONFIGS["1.5b-long"].replace(prompt_len=1024, new_tokens=6)
    model = synth.make_model(shape)
    taus = [0.6, 0.5, 0.4]
    fo, fg, recs, orc, eng = teacher_forced(shape, model, shape.new_tokens, taus, capture=False, persistent=True)
    assert fo == fg
    check_records(recs, taus, capture=False)


def test_1p5b_persistent_agrees_with_five_launch_path():
    """Free-running 1.5B decode: same tokens and gate verdicts on both GPU
    paths; confidences within the parity tolerance."""
    from paper_2609_14144_gb300 import OPT_PERSISTENT, Engine

    shape = synth.CONFIGS["1.5b"].replace(prompt_len=128, new_tokens=32)
    model = synth.make_model(shape)
    outs = []
    for pers in (0, 1):
        eng = Engine(shape, model, max_ctx=shape.prompt_len + shape.new_tokens)
        eng.set_option(OPT_PERSISTENT, pers)
        first = eng.prefill(synth.prompt(shape, shape.prompt_len))
        tok, ex, cf = eng.decode_n(shape.new_tokens, [0.5], input_token=first)
        outs.append((first, tok, ex, cf))
        eng.close()
    (f0, t0, e0, c0), (f1, t1, e1, c1) = outs
    assert f0 == f1
    near = np.abs(c0 - 0.5) < 1e-3
    agree = (t0 == t1) & (e0 == e1)
    # a near-threshold step may go either way; after it the streams may differ
    first_diff = np.argmax(~agree) if not agree.all() else len(agree)
    assert first_diff == len(agree) or near[first_diff]
    assert np.max(np.abs(c0[:first_diff] - c1[:first_diff]), initial=0) < 1e-3


def test_waits_that_run_out_report_a_stall_and_reset_recovers():
    """Failure detection of the persistent layer kernel's bounded waits: with
    the wait bound lowered to 400 SM cycles, ordinary waits (ring stages,
    values from other CTAs) run out.  The launch ends by itself with the
    device error word set, the call reports EE_EDEVICE, and after ee_reset
    with the normal bound the engine decodes like the oracle again."""
    from paper_2609_14144_gb300 import OPT_WAIT_LIMIT, EEError, Engine

    tiny = synth.CONFIGS["tiny"]
    model = synth.make_model(tiny)
    prompt = synth.prompt(tiny)
    eng = Engine(tiny, model)
    assert eng.persistent
    eng.prefill(prompt)
    eng.set_option(OPT_WAIT_LIMIT, 400)
    with pytest.raises(EEError) as e:
        eng.decode_step(int(prompt[-1]), [0.5])
    assert e.value.code == -5 and "timed out" in str(e.value)
    eng.set_option(OPT_WAIT_LIMIT, 0)
    eng.reset()
    orc = oracle.Oracle(tiny, model)
    first = orc.prefill(prompt)
    assert eng.prefill(prompt) == first
    recs = gpu_replay(eng, oracle_steps(orc, first, 12, [0.5]), [0.5], capture=False)
    check_records(recs, [0.5], capture=False)
    eng.close()
