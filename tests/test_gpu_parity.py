"""GPU decode path vs the CPU oracle under teacher forcing (needs a GB300).

The oracle runs free; the GPU engine is driven with the oracle's input tokens
and exit decisions through the C ABI.  On steps outside the exclusion band
(|p - tau| or a top-2 gap below 1e-3) token ids and gate verdicts must match
bit for bit; KV positions (which layer/position was computed or filled) must
match bit for bit; hidden states, logits and KV values within 1e-2 relative
error (max |diff| / max |ref|); confidences within helpers.P_TOL."""
import numpy as np
import pytest

import oracle
import synth
from helpers import P_TOL, check_kv, check_records, is_excluded, rel_err, teacher_forced

pytestmark = pytest.mark.gpu

TINY = synth.CONFIGS["tiny"]


@pytest.fixture(scope="module")
def tiny_model():
    return synth.make_model(TINY)


@pytest.mark.parametrize("tau", [0.5, 0.0, 1.01])
@pytest.mark.parametrize("persistent", [True, False])
def test_tiny_teacher_forced(tiny_model, tau, persistent):
    n = TINY.new_tokens
    fo, fg, recs, orc, eng = teacher_forced(TINY, tiny_model, n, [tau], persistent=persistent)
    assert fo == fg
    excluded = check_records(recs, [tau])
    assert excluded <= n // 8
    check_kv(orc, eng, TINY, TINY.prompt_len + n)
    st, so = eng.stats(), orc.stats()
    assert st["steps"] == so["steps"] == n and st["exits"] == so["exits"] and st["full_steps"] == so["full_steps"]
    if tau == 0.0:
        assert so["exits"] == [n]
    if tau > 1:
        assert so["exits"] == [0]


def test_tiny_eager_path_and_no_pdl_match_graphs(tiny_model):
    n = 24
    _, _, a, _, _ = teacher_forced(TINY, tiny_model, n, [0.5], capture=False)
    _, _, b, _, _ = teacher_forced(TINY, tiny_model, n, [0.5], capture=False, graphs=False)
    _, _, c, _, _ = teacher_forced(TINY, tiny_model, n, [0.5], capture=False, pdl=False)
    for x, y, z in zip(a, b, c):
        assert x["g"] == y["g"] == z["g"]


def test_tiny_permuted_pages(tiny_model):
    n = TINY.new_tokens
    pages = (TINY.max_ctx + 15) // 16
    perm = np.random.default_rng(0).permutation(pages).astype(np.int32)
    fo, fg, recs, orc, eng = teacher_forced(TINY, tiny_model, n, [0.5], page_perm=perm, page_size=16)
    assert fo == fg
    check_records(recs, [0.5])
    check_kv(orc, eng, TINY, TINY.max_ctx)


@pytest.mark.parametrize("prompt_len,n", [(500, 24), (1000, 40)])
def test_tiny_attention_split_geometry_changes(tiny_model, prompt_len, n):
    """16-position pages: past 512 and 1024 positions the pages per attention
    split grow and the split count drops (32 -> 17, 32 -> 22), so split slots
    fall out of use and come back later; their partials must never be taken
    from an earlier layer or launch."""
    shape = TINY.replace(prompt_len=prompt_len)
    prompt = synth.prompt(shape)
    fo, fg, recs, orc, eng = teacher_forced(shape, tiny_model, n, [0.5], prompt=prompt, page_size=16,
                                            capture=False)
    assert fo == fg
    assert check_records(recs, [0.5], capture=False) <= n // 8
    for j in (0, TINY.n_layers - 1):
        for t in range(prompt_len - 4, prompt_len + n):
            ko, vo, so = orc.kv(j, t)
            kg, vg = eng.kv(j, t)
            assert eng.kv_src(j, t) == so
            assert rel_err(kg, ko) <= 1e-2 and rel_err(vg, vo) <= 1e-2, (j, t)


def test_tiny_bias_and_tied_head():
    shape = TINY.replace(qkv_bias=True, tied_embedding=True, new_tokens=24)
    model = synth.make_model(shape)
    fo, fg, recs, orc, eng = teacher_forced(shape, model, shape.new_tokens, [0.5])
    assert fo == fg
    check_records(recs, [0.5])
    check_kv(orc, eng, shape, shape.max_ctx)


def test_tiny_three_readouts():
    shape = TINY.replace(readout_layers=(1, 2, 3), new_tokens=48)
    model = synth.make_model(shape)
    taus = [0.7, 0.5, 0.4]
    fo, fg, recs, orc, eng = teacher_forced(shape, model, shape.new_tokens, taus)
    assert fo == fg
    check_records(recs, taus)
    check_kv(orc, eng, shape, shape.max_ctx)
    assert len({r["o"]["exit_readout"] for r in recs}) >= 3  # several outcomes exercised


def test_tiny_decode_n_free_run_matches_oracle(tiny_model):
    """ee_decode_n (WHILE-node graph, token fed back on the device) against
    the oracle's free run, up to the first step inside the exclusion band."""
    from paper_2609_14144_gb300 import Engine

    n, taus = TINY.new_tokens, [0.5]
    orc = oracle.Oracle(TINY, tiny_model)
    first, ref = orc.generate(synth.prompt(TINY), n, taus)
    eng = Engine(TINY, tiny_model)
    assert eng.prefill(synth.prompt(TINY)) == first
    tok, ex, cf = eng.decode_n(n, taus)
    for i, r in enumerate(ref):
        if is_excluded(r, taus):
            break
        assert tok[i] == r["token"] and ex[i] == r["exit_readout"], i
        assert abs(cf[i] - r["confidence"][0]) <= P_TOL
    st = eng.stats()
    assert st["steps"] == n and eng.position == TINY.max_ctx


def test_tiny_decode_n_split_calls_and_device_outputs(tiny_model):
    """Two decode_n calls equal one; device-side outputs equal host outputs."""
    import torch

    from paper_2609_14144_gb300 import DEVICE, Engine

    taus = [0.5]
    a = Engine(TINY, tiny_model)
    a.prefill(synth.prompt(TINY))
    t1, e1, _ = a.decode_n(40, taus)
    b = Engine(TINY, tiny_model)
    b.prefill(synth.prompt(TINY))
    t2a, e2a, _ = b.decode_n(17, taus)
    tt, ee, cc = b.decode_n(23, taus, where=DEVICE)
    b.sync()
    assert np.array_equal(t1, np.concatenate([t2a, tt.cpu().numpy()]))
    assert np.array_equal(e1, np.concatenate([e2a, ee.cpu().numpy()]))
    assert a.stats() == b.stats()
    del torch


def test_tiny_imposed_exit_schedule(tiny_model):
    """Imposed exits (the paper's timing method, App. C): the schedule, not the
    gate, decides; the oracle with the same schedule agrees."""
    from paper_2609_14144_gb300 import FORCE_EXIT_AT, FORCE_FULL, Engine

    n = TINY.new_tokens
    sched = np.where(synth.exit_schedule(TINY, n, 0.5) == 1, FORCE_EXIT_AT(0), FORCE_FULL).astype(np.int8)
    orc = oracle.Oracle(TINY, tiny_model)
    first, ref = orc.generate(synth.prompt(TINY), n, [0.5], force_schedule=sched)
    eng = Engine(TINY, tiny_model)
    eng.prefill(synth.prompt(TINY))
    tok, ex, _ = eng.decode_n(n, [0.5], schedule=sched)
    assert np.array_equal(ex, np.where(sched == FORCE_FULL, -1, 0))
    for i, r in enumerate(ref):
        if is_excluded(r, [2.0]) or (r["exited"] and r["gap"][0] < 1e-3):
            break
        assert tok[i] == r["token"], i


def test_gpu_invariants_tau(tiny_model):
    """tau > 1 gives exactly the plain model's tokens (no readout attached);
    tau = 0 exits every step."""
    from paper_2609_14144_gb300 import Engine

    n = TINY.new_tokens
    plain = Engine(TINY, tiny_model, readouts=False)
    first = plain.prefill(synth.prompt(TINY))
    tp, ep, _ = plain.decode_n(n)
    gated = Engine(TINY, tiny_model)
    assert gated.prefill(synth.prompt(TINY)) == first
    tg, eg, _ = gated.decode_n(n, [1.01])
    assert np.array_equal(tp, tg) and (eg == -1).all() and (ep == -1).all()
    always = Engine(TINY, tiny_model)
    always.prefill(synth.prompt(TINY))
    _, ea, _ = always.decode_n(n, [0.0])
    assert (ea == 0).all() and always.stats()["exits"] == [n]


def test_api_errors(tiny_model):
    from paper_2609_14144_gb300 import EEError, Engine

    eng = Engine(TINY, tiny_model)
    with pytest.raises(EEError) as e:
        eng.decode_step(1, [0.5])
    assert e.value.code == -6  # before prefill
    with pytest.raises(EEError) as e:
        eng.prefill([0, TINY.vocab])
    assert e.value.code == -1
    with pytest.raises(EEError) as e:
        eng.prefill([])  # an empty prompt
    assert e.value.code == -1
    eng.prefill(synth.prompt(TINY))
    with pytest.raises(EEError) as e:
        eng.decode_step(TINY.vocab, [0.5])
    assert e.value.code == -1
    with pytest.raises(EEError) as e:
        eng.decode_n(TINY.new_tokens + 1, [0.5])
    assert e.value.code == -4
    with pytest.raises(EEError) as e:
        eng.add_readout(3, tiny_model["readouts"][0][1], tiny_model["readouts"][0][2])
    assert e.value.code == -6
    eng.decode_n(TINY.new_tokens, [0.5])
    with pytest.raises(EEError) as e:
        eng.decode_step(-1, [0.5])
    assert e.value.code == -4
    eng.reset()
    assert eng.position == 0
    eng.prefill(synth.prompt(TINY))


def test_tiny_prompt_of_max_ctx_positions(tiny_model):
    """The largest prompt a context holds (max_ctx positions, two batches of
    the multi-position pass with a ragged tail): first token as the oracle's,
    and the next step is refused (no room for its position)."""
    from paper_2609_14144_gb300 import EEError, Engine

    n = 150
    prompt = synth.token_ids(TINY.seed, 907, n, TINY.vocab)
    orc = oracle.Oracle(TINY, tiny_model, max_ctx=n)
    tok_o, cap = orc.prefill(prompt, capture=True)
    eng = Engine(TINY, tiny_model, max_ctx=n)
    tok_g = eng.prefill(prompt)
    z = np.sort(np.asarray(cap["final_logits"], np.float64))
    p = np.exp(z - z[-1])
    if (p[-1] - p[-2]) / p.sum() >= 1e-3:
        assert tok_g == tok_o
    with pytest.raises(EEError) as e:
        eng.decode_step(tok_g, [0.5])
    assert e.value.code == -4
    eng.close()


def test_half_b_teacher_forced():
    """0.5B shape (d 896, 14/2 heads of 64, F 4864, V 151936), short prompt."""
    shape = synth.CONFIGS["0.5b"].replace(prompt_len=48, new_tokens=12)
    model = synth.make_model(shape)
    fo, fg, recs, orc, eng = teacher_forced(shape, model, shape.new_tokens, [0.5])
    assert fo == fg
    check_records(recs, [0.5])
    check_kv(orc, eng, shape, shape.max_ctx)


def test_1p5b_teacher_forced_bench_config():
    """1.5B shape at the benchmark's prompt length (512) and launch setup."""
    shape = synth.CONFIGS["1.5b"].replace(new_tokens=6)
    model = synth.make_model(shape)
    fo, fg, recs, orc, eng = teacher_forced(shape, model, shape.new_tokens, [0.5])
    assert fo == fg
    check_records(recs, [0.5])
    for j in (0, 13, 14, 27):
        for t in (0, 255, 511, 512, shape.max_ctx - 1):
            ko, vo, so = orc.kv(j, t)
            assert eng.kv_src(j, t) == so


def test_1p5b_long_three_readouts_structure():
    """The long-context three-readout shape (readouts 7, 14, 21), prompt cut to
    1024 positions so the oracle finishes in seconds."""
    shape = synth.CONFIGS["1.5b-long"].replace(prompt_len=1024, new_tokens=6)
    model = synth.make_model(shape)
    taus = [0.6, 0.5, 0.4]
    fo, fg, recs, orc, eng = teacher_forced(shape, model, shape.new_tokens, taus, capture=False)
    assert fo == fg
    check_records(recs, taus, capture=False)


@pytest.mark.parametrize("kind,tau", [(1, 0.25), (2, -2.0)])
@pytest.mark.parametrize("persistent", [True, False])
def test_tiny_margin_and_entropy_gates(tiny_model, kind, tau, persistent):
    """Section 10: the gate on the margin p1 - p2 or on the negative entropy;
    tokens, verdicts and recorded signals against the oracle's."""
    n = TINY.new_tokens
    fo, fg, recs, orc, eng = teacher_forced(TINY, tiny_model, n, [tau], conf_kind=kind, persistent=persistent)
    assert fo == fg
    excluded = check_records(recs, [tau])
    assert excluded <= n // 8
    st, so = eng.stats(), orc.stats()
    assert 0 < so["exits"][0] < n
    assert st["exits"] == so["exits"]


def test_1p5b_entropy_gate():
    shape = synth.CONFIGS["1.5b"].replace(new_tokens=6)
    model = synth.make_model(shape)
    fo, fg, recs, orc, eng = teacher_forced(shape, model, shape.new_tokens, [-3.0], conf_kind=2)
    assert fo == fg
    check_records(recs, [-3.0])
