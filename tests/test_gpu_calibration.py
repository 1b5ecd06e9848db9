"""Fidelity calibration on the GPU against the oracle (needs a GB300).

Section 2 accepts an early answer when its token lies in the full model's
nucleus (the smallest most-probable set holding 90 percent of the mass);
Section 4, step four picks the lowest tau at which at least 90 percent of the
early answers are acceptable.  The engine's calibration pass runs teacher-
forced full-depth steps in one graph launch and records every readout's
confidence with readout 0's nucleus membership; the threshold selection runs
on the device.  Both are compared with the oracle: confidences within 1e-3,
membership bit for bit outside the band where the oracle's mass sits within
rounding of the nucleus share, masses within 2e-3, thresholds exactly on
identical inputs."""
import math

import numpy as np
import pytest
import torch

import oracle
import synth
from helpers import (EXCLUDE_EPS, MASS_TOL, P_TOL, check_kv, damped_after_readout, is_excluded, nucleus_ambiguity,
                     teacher_forced)

pytestmark = pytest.mark.gpu

TINY = synth.CONFIGS["tiny"]


@pytest.fixture(scope="module")
def near_model():
    """The tiny shape with the layers after the readout silenced: a mix of
    acceptable and unacceptable early answers."""
    return damped_after_readout(TINY, synth.make_model(TINY), 0.0)


def oracle_pass(shape, model, prompt, ids, p_nuc, conf_kind=0):
    R = len(shape.readout_layers)
    orc = oracle.Oracle(shape, model, max_ctx=len(prompt) + len(ids) + 1)
    orc.set_confidence(conf_kind)
    orc.set_nucleus(p_nuc)
    orc.prefill(prompt)
    recs = [orc.decode_step(int(t), [2.0] * R, oracle.FORCE_FULL, capture=True) for t in ids]
    return orc, recs


def check_calibration(recs, conf, member, mass, p_nuc):
    """Assert the parity rules; returns the number of excluded steps."""
    excluded = 0
    for i, o in enumerate(recs):
        assert o["nucleus_member"] in (0, 1)
        for r in range(o["n_evaluated"]):
            assert abs(conf[i, r] - o["confidence"][r]) <= P_TOL, (i, r, conf[i], o["confidence"])
        amb, bound = nucleus_ambiguity(o["capture"]["final_logits"], o["readout_token"][0], p_nuc, o["nucleus_mass"])
        if o["gap"][0] < EXCLUDE_EPS or amb:
            excluded += 1
            continue
        assert member[i] == o["nucleus_member"], (i, member[i], o["nucleus_mass"], mass[i])
        assert abs(mass[i] - o["nucleus_mass"]) <= MASS_TOL + bound, (i, mass[i], o["nucleus_mass"], bound)
    return excluded


@pytest.mark.parametrize("persistent", [True, False])
@pytest.mark.parametrize("graphs", [True, False])
def test_tiny_calibrate_matches_oracle(near_model, persistent, graphs):
    from paper_2609_14144_gb300 import FORCE_FULL, OPT_GRAPHS, OPT_PERSISTENT, Engine

    n, p_nuc = 48, 0.9
    prompt = synth.prompt(TINY)
    ids = synth.calibration_stream(TINY, n)
    orc, recs = oracle_pass(TINY, near_model, prompt, ids, p_nuc)
    eng = Engine(TINY, near_model, max_ctx=len(prompt) + n + 1)
    eng.set_option(OPT_PERSISTENT, int(persistent))
    eng.set_option(OPT_GRAPHS, int(graphs))
    eng.prefill(prompt)
    conf, member, mass = eng.calibrate(ids, p_nuc)
    assert conf.shape == (n, 1) and member.shape == (n,) and mass.shape == (n,)
    excluded = check_calibration(recs, conf, member, mass, p_nuc)
    assert excluded <= n // 8
    om = np.array([o["nucleus_member"] for o in recs])
    assert 0 < om.sum() < n, "the workload should hold both outcomes"
    # the pass leaves the full model's cache and position behind it
    assert eng.position == len(prompt) + n
    st = eng.stats()
    assert st["steps"] == n and st["full_steps"] == n and st["exits"] == [0]
    check_kv(orc, eng, TINY, len(prompt) + n)
    # the next input is the full model's token after the last id
    o = orc.decode_step(recs[-1]["token"], [2.0], oracle.FORCE_FULL)
    g = eng.decode_step(-1, [2.0], FORCE_FULL)
    if not is_excluded(recs[-1], [2.0]) and not is_excluded(o, [2.0]):
        assert g["token"] == o["token"]


def test_tiny_calibrate_device_arrays_match_host(near_model):
    from paper_2609_14144_gb300 import DEVICE, Engine

    n = 40
    prompt = synth.prompt(TINY)
    ids = synth.calibration_stream(TINY, n)
    eng = Engine(TINY, near_model, max_ctx=len(prompt) + n)
    eng.prefill(prompt)
    ch, mh, sh = eng.calibrate(ids, 0.8)
    eng.reset()
    eng.prefill(prompt)
    d_ids = torch.from_numpy(np.asarray(ids, np.int32)).to(eng.device)
    torch.cuda.synchronize()
    cd, md, sd = eng.calibrate(d_ids, 0.8, where=DEVICE)
    eng.sync()
    assert np.array_equal(cd.cpu().numpy(), ch)
    assert np.array_equal(md.cpu().numpy(), mh)
    assert np.array_equal(sd.cpu().numpy(), sh)
    # the share moves the verdicts, not the masses
    assert np.array_equal(mh, (sh < np.float32(0.8)).astype(np.int32))


def test_tiny_calibrate_three_readouts_and_signals():
    """Every readout's signal is recorded (margin and negative entropy too);
    membership stays readout 0's."""
    from paper_2609_14144_gb300 import OPT_CONFIDENCE, Engine

    shape = TINY.replace(n_layers=6, readout_layers=(1, 2, 4))
    model = damped_after_readout(shape, synth.make_model(shape), 0.0)
    n, p_nuc = 24, 0.9
    prompt = synth.prompt(shape)
    ids = synth.calibration_stream(shape, n)
    for kind in (0, 1, 2):
        orc, recs = oracle_pass(shape, model, prompt, ids, p_nuc, conf_kind=kind)
        eng = Engine(shape, model, max_ctx=len(prompt) + n)
        eng.set_option(OPT_CONFIDENCE, kind)
        eng.prefill(prompt)
        conf, member, mass = eng.calibrate(ids, p_nuc)
        assert conf.shape == (n, 3)
        assert check_calibration(recs, conf, member, mass, p_nuc) <= n // 8
        eng.close()


@pytest.mark.parametrize("persistent", [True, False])
def test_tiny_decode_step_reports_nucleus(near_model, persistent):
    """EE_OPT_NUCLEUS: gated steps report readout 0's membership on full
    steps and -1 on exit steps."""
    n, tau = 32, 0.6
    fo, fg, recs, orc, eng = teacher_forced(TINY, near_model, n, [tau], persistent=persistent,
                                            nucleus_permille=900)
    assert fo == fg
    exits = fulls = 0
    for i, rec in enumerate(recs):
        o, g = rec["o"], rec["g"]
        if o["exited"]:
            exits += 1
            assert g["nucleus_member"] == -1 and o["nucleus_member"] == -1
            continue
        fulls += 1
        amb, bound = nucleus_ambiguity(o["capture"]["final_logits"], o["readout_token"][0], 0.9, o["nucleus_mass"])
        if amb or is_excluded(o, [tau]):
            continue
        assert g["nucleus_member"] == o["nucleus_member"], i
        assert abs(g["nucleus_mass"] - o["nucleus_mass"]) <= MASS_TOL + bound, i
    assert exits > 0 and fulls > 0


def test_select_tau_matches_oracle():
    from paper_2609_14144_gb300 import select_tau

    rng = np.random.default_rng(11)
    for n in (1, 2, 7, 300, 2047, 20000):
        for levels in (None, 5):
            conf = rng.random(n).astype(np.float32)
            if levels:
                conf = (np.floor(conf * levels) / levels).astype(np.float32)  # ties
            member = (rng.random(n) < 0.3 + 0.7 * conf).astype(np.int32)
            dc, dm = torch.from_numpy(conf).cuda(), torch.from_numpy(member).cuda()
            for target in (0.0, 0.5, 0.9, 0.97, 1.0):
                t = np.float32(target)
                got = select_tau(dc, dm, float(t)).item()
                want = oracle.select_tau(conf, member, float(t))
                assert got == want or (math.isinf(got) and math.isinf(want) and got == want), (n, levels, target)


def test_select_tau_strided_column_and_edges():
    from paper_2609_14144_gb300 import select_tau

    rng = np.random.default_rng(12)
    n = 3000
    table = rng.random((n, 3)).astype(np.float32)
    member = (rng.random(n) < table[:, 1]).astype(np.int32)
    dt, dm = torch.from_numpy(table).cuda(), torch.from_numpy(member).cuda()
    got = select_tau(dt[:, 1], dm, 0.9).item()
    assert got == oracle.select_tau(np.ascontiguousarray(table[:, 1]), member, 0.9)
    conf = torch.from_numpy(table[:, 0].copy()).cuda()
    assert select_tau(conf, torch.ones(n, dtype=torch.int32, device="cuda"), 0.9).item() == -math.inf
    assert select_tau(conf, torch.zeros(n, dtype=torch.int32, device="cuda"), 0.9).item() == math.inf
    # acceptability rising with confidence: tau sits below the acceptable run
    c = torch.arange(10, dtype=torch.float32, device="cuda") / 10
    m = torch.tensor([0, 0, 0, 1, 0, 1, 1, 1, 1, 1], dtype=torch.int32, device="cuda")
    assert select_tau(c, m, 1.0).item() == np.float32(0.4)
    assert select_tau(c, m, 0.8).item() == np.float32(0.2)


def test_select_tau_large_grid_against_sorted_counts():
    """More candidates than one pass of the grid holds: checked against the
    counts of every candidate taken from a sort."""
    from paper_2609_14144_gb300 import select_tau

    rng = np.random.default_rng(13)
    n = 200_000
    conf = rng.random(n).astype(np.float32)
    member = (rng.random(n) < 0.6 + 0.4 * conf).astype(np.int32)
    target = 0.93
    got = select_tau(torch.from_numpy(conf).cuda(), torch.from_numpy(member).cuda(), target).item()
    order = np.argsort(conf, kind="stable")
    cs = conf[order]
    good_suffix = np.concatenate([np.cumsum(member[order][::-1])[::-1], [0]])
    cands = np.concatenate([[-np.inf], np.unique(cs)])
    first_above = np.searchsorted(cs, cands, side="right")
    early = n - first_above
    good = good_suffix[first_above]
    ok = (early > 0) & (good >= np.float64(np.float32(target)) * early)
    want = cands[ok].min() if ok.any() else np.inf
    assert got == np.float32(want)


def test_calibrate_then_select_matches_oracle_pipeline(near_model):
    """The on-device pipeline (calibration pass, then threshold selection on
    its device outputs) against the oracle's."""
    from paper_2609_14144_gb300 import DEVICE, Engine, select_tau

    n, p_nuc, target = 64, 0.9, 0.9
    prompt = synth.prompt(TINY)
    ids = synth.calibration_stream(TINY, n)
    orc, recs = oracle_pass(TINY, near_model, prompt, ids, p_nuc)
    eng = Engine(TINY, near_model, max_ctx=len(prompt) + n)
    eng.prefill(prompt)
    d_ids = torch.from_numpy(np.asarray(ids, np.int32)).to(eng.device)
    torch.cuda.synchronize()
    conf, member, mass = eng.calibrate(d_ids, p_nuc, where=DEVICE)
    t = select_tau(conf[:, 0], member, target, stream=eng.stream)
    eng.sync()
    tau = t.item()
    # identical inputs: identical threshold
    c_h, m_h = conf[:, 0].cpu().numpy().copy(), member.cpu().numpy()
    assert tau == oracle.select_tau(c_h, m_h, target)
    # against the oracle's own pass
    oc = np.array([o["confidence"][0] for o in recs], np.float32)
    om = np.array([o["nucleus_member"] for o in recs], np.int32)
    check_calibration(recs, conf.cpu().numpy(), m_h, mass.cpu().numpy(), p_nuc)
    if np.array_equal(m_h, om):
        tau_o = oracle.select_tau(oc, om, target)
        assert (math.isinf(tau) and tau == tau_o) or abs(tau - tau_o) <= P_TOL
    assert math.isfinite(tau), "the workload should admit a finite threshold"


def test_1p5b_calibrate_sampled():
    """The 1.5B shape at the benchmark's prompt length: a short calibration
    pass against the oracle."""
    from paper_2609_14144_gb300 import Engine

    shape = synth.CONFIGS["1.5b"]
    model = synth.make_model(shape)
    n, p_nuc = 8, 0.9
    prompt = synth.prompt(shape)
    ids = synth.calibration_stream(shape, n)
    orc, recs = oracle_pass(shape, model, prompt, ids, p_nuc)
    eng = Engine(shape, model, max_ctx=len(prompt) + n)
    eng.prefill(prompt)
    conf, member, mass = eng.calibrate(ids, p_nuc)
    assert check_calibration(recs, conf, member, mass, p_nuc) <= 1
    assert eng.position == len(prompt) + n


def test_calibration_api_errors(near_model):
    from paper_2609_14144_gb300 import EEError, Engine, select_tau

    prompt = synth.prompt(TINY)
    eng = Engine(TINY, near_model, max_ctx=len(prompt) + 8)
    with pytest.raises(EEError):
        eng.calibrate([1, 2, 3])  # before prefill
    eng.prefill(prompt)
    for bad in (dict(ids=[]), dict(ids=[1, 2], p_nuc=0.0), dict(ids=[1, 2], p_nuc=1.5),
                dict(ids=[1, TINY.vocab]), dict(ids=[1] * 9)):
        with pytest.raises(EEError):
            eng.calibrate(**bad)
    assert eng.position == len(prompt)
    conf, member, mass = eng.calibrate([1, 2, 3])
    assert conf.shape == (3, 1) and eng.position == len(prompt) + 3
    plain = Engine(TINY, near_model, max_ctx=len(prompt) + 8, readouts=False)
    plain.prefill(prompt)
    with pytest.raises(EEError):
        plain.calibrate([1, 2])
    c = torch.zeros(4, device="cuda")
    m = torch.zeros(4, dtype=torch.int32, device="cuda")
    with pytest.raises(EEError):
        select_tau(c, m, 1.5)
    with pytest.raises(EEError):
        select_tau(c[:0], m[:0], 0.9)
