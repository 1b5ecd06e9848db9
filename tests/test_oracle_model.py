"""Model-level pins of the oracle (no GPU): the invariants the paper's
definitions fix, and special weight settings whose result has a closed form."""
import math

import numpy as np
import pytest
import scipy.special

import oracle
import synth
from helpers import bf16_round, identity_bits, micro, one_hot_matrix, to_bf16_bits, zeros_like_bits

TINY = synth.CONFIGS["tiny"]


def _run(shape, model, taus, n=None, readouts=True, force=None):
    o = oracle.Oracle(shape, model, readouts=readouts)
    first, steps = o.generate(synth.prompt(shape), n or shape.new_tokens, taus, force_schedule=force)
    return o, first, steps


# ------------------------------------------------------------- I-1
def test_tau_above_one_reproduces_the_plain_model():
    """Section 2 / Section 4 step five: a gate that never passes leaves the
    full model's greedy output untouched."""
    model = synth.make_model(TINY)
    og, first_g, gated = _run(TINY, model, [1.01])
    op, first_p, plain = _run(TINY, model, [], readouts=False)
    assert first_g == first_p
    assert [s["token"] for s in gated] == [s["token"] for s in plain]
    assert all(not s["exited"] for s in gated) and og.stats()["exits"] == [0]
    for j in range(TINY.n_layers):
        for t in (0, TINY.prompt_len, TINY.max_ctx - 1):
            kg, vg, sg = og.kv(j, t)
            kp, vp, sp = op.kv(j, t)
            assert np.array_equal(kg, kp) and np.array_equal(vg, vp) and sg == sp == 1


# ------------------------------------------------------------- I-2
def test_tau_zero_always_exits_and_never_reads_upper_layer_q_o_ffn():
    """tau = 0 exits every step at layer k (p >= 1/V > 0); the upper layers'
    query, output and FFN weights are then never read, so editing them after
    prefill changes nothing."""
    shape = TINY
    k = shape.readout_layers[0]
    ref_model = synth.make_model(shape)
    o_ref, f_ref, s_ref = _run(shape, ref_model, [0.0])
    edit = synth.make_model(shape)
    o = oracle.Oracle(shape, edit)
    first = o.prefill(synth.prompt(shape))
    rng = np.random.default_rng(5)
    for j in range(k, shape.n_layers):
        for key in ("wq", "wo", "wg", "wu", "wd"):
            edit["layers"][j][key][...] = rng.integers(0, 65535, edit["layers"][j][key].shape, dtype=np.uint16)
    tok, steps = first, []
    for _ in range(shape.new_tokens):
        s = o.decode_step(tok, [0.0])
        steps.append(s)
        tok = s["token"]
    assert first == f_ref
    assert all(s["exited"] and s["exit_layer"] == k for s in steps)
    assert [s["token"] for s in steps] == [s["token"] for s in s_ref]
    assert [s["confidence"] for s in steps] == [s["confidence"] for s in s_ref]
    assert o.stats()["exits"] == [shape.new_tokens]
    assert all(s["token"] == s["readout_token"][0] for s in steps)
    for j in range(shape.n_layers):
        for t in range(shape.prompt_len, shape.max_ctx):
            assert o.kv(j, t)[2] == (2 if j >= k else 1)


# ------------------------------------------------------------- I-3
def _with_identity_readout_at_L(shape, model):
    d = shape.d_model
    model = dict(model)
    model["readouts"] = [(shape.n_layers, identity_bits(d), zeros_like_bits(np.zeros(d)))]
    return shape.replace(readout_layers=(shape.n_layers,)), model


def test_identity_readout_at_last_layer_reproduces_final_logits():
    """Section 2: the readout's output passes through the model's own final
    normalisation and unembedding unchanged, so an identity readout at layer L
    gives the final logits bit for bit (fp32 activations)."""
    shape, model = _with_identity_readout_at_L(micro(), synth.make_model(micro()))
    o = oracle.Oracle(shape, model)
    tok = o.prefill(synth.prompt(shape))
    for _ in range(6):
        s = o.decode_step(tok, [1.01], capture=True)
        cap = s["capture"]
        assert np.array_equal(cap["readout_logits"][0], cap["final_logits"])
        assert s["readout_token"][0] == s["full_token"]
        tok = s["token"]
    # with bf16 activations the readout input is bf16(h): logits agree to 1e-2
    o2 = oracle.Oracle(shape, model, bf16_activations=True)
    tok = o2.prefill(synth.prompt(shape))
    for _ in range(6):
        s = o2.decode_step(tok, [1.01], capture=True)
        r, f = s["capture"]["readout_logits"][0], s["capture"]["final_logits"]
        assert np.max(np.abs(r - f)) <= 1e-2 * np.max(np.abs(f))
        tok = s["token"]


def test_identity_readout_tau_zero_equals_tau_above_one():
    shape, model = _with_identity_readout_at_L(micro(), synth.make_model(micro()))
    _, f1, a = _run(shape, model, [0.0])
    _, f2, b = _run(shape, model, [1.01])
    assert f1 == f2 and [s["token"] for s in a] == [s["token"] for s in b]
    assert all(s["exited"] for s in a) and not any(s["exited"] for s in b)


# ------------------------------------------------------------- I-4
def test_kv_fill_equals_full_path_when_upper_layers_leave_the_residual_unchanged():
    """Section 4 step five: the fill projects the exit-layer state through the
    skipped layers' key/value matrices.  If those layers add nothing to the
    residual (zero output and down projections) the full path computes exactly
    the same keys and values."""
    shape = micro()
    k = shape.readout_layers[0]
    model = synth.make_model(shape)
    for j in range(k, shape.n_layers):
        model["layers"][j]["wo"] = zeros_like_bits(model["layers"][j]["wo"])
        model["layers"][j]["wd"] = zeros_like_bits(model["layers"][j]["wd"])
    full = oracle.Oracle(shape, model)
    ex = oracle.Oracle(shape, model)
    tok = full.prefill(synth.prompt(shape))
    assert ex.prefill(synth.prompt(shape)) == tok
    for _ in range(shape.new_tokens):
        a = full.decode_step(tok, [0.5], oracle.FORCE_FULL)
        b = ex.decode_step(tok, [0.5], oracle.FORCE_EXIT_AT(0))
        t = full.pos - 1
        for j in range(shape.n_layers):
            ka, va, sa = full.kv(j, t)
            kb, vb, sb = ex.kv(j, t)
            assert np.array_equal(ka, kb) and np.array_equal(va, vb)
            assert sa == 1 and sb == (2 if j >= k else 1)
        assert a["confidence"] == b["confidence"]
        tok = a["token"]


# ------------------------------------------------------------- multi-exit
def test_multiple_readouts_shallowest_passing_exits():
    """Section 4 step three: several exit points; the first passing one is taken
    and every layer above it is filled."""
    shape = micro(readout_layers=(1, 2, 3))
    model = synth.make_model(shape)
    cases = [([1.01, 0.0, 0.0], 1), ([0.0, 0.0, 0.0], 0), ([1.01, 1.01, 0.0], 2), ([1.01] * 3, None)]
    for taus, expect in cases:
        o, _, steps = _run(shape, model, taus, n=4)
        for s in steps:
            if expect is None:
                assert not s["exited"] and s["n_evaluated"] == 3 and s["exit_layer"] == shape.n_layers
            else:
                assert s["exited"] and s["exit_readout"] == expect and s["n_evaluated"] == expect + 1
                assert s["exit_layer"] == shape.readout_layers[expect]
        e_layer = shape.n_layers if expect is None else shape.readout_layers[expect]
        for j in range(shape.n_layers):
            assert o.kv(j, shape.prompt_len + 1)[2] == (1 if j < e_layer else 2)
    # forced exit at the last readout still reports the earlier gates' verdicts
    o = oracle.Oracle(shape, model)
    tok = o.prefill(synth.prompt(shape))
    s = o.decode_step(tok, [0.0, 0.0, 0.0], oracle.FORCE_EXIT_AT(2))
    assert s["exit_readout"] == 2 and s["gate_pass"] == [1, 1, 1] and s["n_evaluated"] == 3


# ------------------------------------------------------------- I-6
def test_exit_count_non_increasing_in_tau():
    model = synth.make_model(TINY)
    _, _, steps = _run(TINY, model, [0.5], force=[oracle.FORCE_FULL] * TINY.new_tokens)
    p = np.array([s["confidence"][0] for s in steps], np.float32)
    taus = np.linspace(0, 1.01, 50).astype(np.float32)
    counts = [int(np.sum(p > t)) for t in taus]
    assert counts[0] == len(p) and counts[-1] == 0
    assert all(a >= b for a, b in zip(counts, counts[1:]))
    # the free gate agrees with its recorded confidence
    for t in (0.3, 0.6):
        _, _, free = _run(TINY, model, [t])
        assert all(s["exited"] == (s["confidence"][0] > np.float32(t)) for s in free)


def test_gate_is_strict():
    """Section 2: the early answer is accepted when its probability exceeds the
    threshold; a threshold equal to the probability does not pass."""
    model = synth.make_model(TINY)
    o = oracle.Oracle(TINY, model)
    tok = o.prefill(synth.prompt(TINY))
    s0 = o.decode_step(tok, [0.5], oracle.FORCE_FULL)
    p = np.float32(s0["confidence"][0])
    for tau, expect in ((p, 0), (np.nextafter(p, np.float32(-1)), 1), (np.float32(1.0), 0)):
        o2 = oracle.Oracle(TINY, model)
        o2.prefill(synth.prompt(TINY))
        s = o2.decode_step(tok, [tau], oracle.FORCE_FULL)
        assert s["confidence"][0] == p and s["gate_pass"][0] == expect


def test_gate_with_margin_and_negative_entropy():
    """Section 10: the gate may compare the margin p1 - p2 or the negative
    entropy with tau instead of p1; the recorded confidence is that signal
    of the readout's distribution, and the gate is still strict."""
    model = synth.make_model(TINY)
    for kind, key in ((oracle.CONF_MARGIN, "gap"), (oracle.CONF_NEGENT, "neg_entropy")):
        o = oracle.Oracle(TINY, model)
        o.set_confidence(kind)
        tok = o.prefill(synth.prompt(TINY))
        sigs = []
        for _ in range(12):
            s = o.decode_step(tok, [0.5], oracle.FORCE_FULL, capture=True)
            c = oracle.confidence(s["capture"]["readout_logits"][0])
            assert s["confidence"][0] == np.float32(c[key])
            assert s["gate_pass"][0] == int(np.float32(c[key]) > np.float32(0.5))
            sigs.append(s["confidence"][0])
            tok = s["token"]
        sigs = np.array(sigs, np.float32)
        if kind == oracle.CONF_MARGIN:
            assert np.all((0.0 <= sigs) & (sigs < 1.0))
        else:
            assert np.all((-math.log(TINY.vocab) - 1e-4 <= sigs) & (sigs <= 0.0))
    # always / never exit at thresholds below and above the signal's range
    for kind, lo, hi in ((oracle.CONF_MARGIN, -0.5, 1.0), (oracle.CONF_NEGENT, -math.log(TINY.vocab) - 1.0, 0.0)):
        for tau, expect in ((lo, TINY.new_tokens), (hi, 0)):
            o = oracle.Oracle(TINY, model)
            o.set_confidence(kind)
            o.generate(synth.prompt(TINY), TINY.new_tokens, [tau])
            assert o.stats()["exits"] == [expect]
    with pytest.raises(ValueError):
        oracle.Oracle(TINY, model).set_confidence(3)


def test_nucleus_membership_of_the_readout_answer():
    """Section 2 acceptance: on full steps the oracle reports whether readout
    0's token lies in the full model's nucleus (from the final logits); on
    exit steps it is not computed."""
    model = synth.make_model(TINY)
    o = oracle.Oracle(TINY, model)
    tok = o.prefill(synth.prompt(TINY))
    seen = set()
    for i in range(24):
        force = oracle.FORCE_EXIT_AT(0) if i % 4 == 3 else oracle.FORCE_FULL
        s = o.decode_step(tok, [0.5], force, capture=True)
        if s["exited"]:
            assert s["nucleus_member"] == -1
        else:
            m, mass = oracle.nucleus_member(s["capture"]["final_logits"], s["readout_token"][0], 0.9)
            assert s["nucleus_member"] == int(m) and s["nucleus_mass"] == np.float32(mass)
            seen.add(s["nucleus_member"])
        tok = s["token"]
    o.set_nucleus(1.0)
    s = o.decode_step(tok, [0.5], oracle.FORCE_FULL)
    assert s["nucleus_member"] == 1
    with pytest.raises(ValueError):
        o.set_nucleus(0.0)


def _exit_run(shape, model, n, every=3, extra=0):
    """Decode n steps with exits imposed at readout 0 on all but every
    `every`-th step; returns (oracle, input tokens of the steps)."""
    o = oracle.Oracle(shape, model, max_ctx=shape.prompt_len + n + extra)
    tok = o.prefill(synth.prompt(shape))
    ins = []
    for i in range(n):
        ins.append(tok)
        s = o.decode_step(tok, [2.0], oracle.FORCE_FULL if i % every == 0 else oracle.FORCE_EXIT_AT(0))
        tok = s["token"]
    return o, ins


def _cache(o, shape, t0, t1):
    return [[o.kv(j, t) for t in range(t0, t1)] for j in range(shape.n_layers)]


def test_repass_reproduces_the_full_depth_cache():
    """Section 11: re-passing every exited position, in order, recomputes
    the cache the full model would hold for the same tokens, bit for bit."""
    n = 20
    model = synth.make_model(TINY)
    o, ins = _exit_run(TINY, model, n)
    P = TINY.prompt_len
    assert o.repass(P, P + n) == n - len(range(0, n, 3))
    full = oracle.Oracle(TINY, model, max_ctx=P + n)
    full.prefill(synth.prompt(TINY))
    for tok in ins:
        full.decode_step(tok, [2.0], oracle.FORCE_FULL)
    for j in range(TINY.n_layers):
        for t in range(P + n):
            ko, vo, so = o.kv(j, t)
            kf, vf, sf = full.kv(j, t)
            assert so == sf == 1, (j, t, so, sf)
            assert np.array_equal(ko, kf) and np.array_equal(vo, vf), (j, t)
    assert o.repass(P, P + n) == 0  # nothing left to re-pass


def test_repass_of_a_range_changes_only_that_range():
    n = 24
    model = synth.make_model(TINY)
    o, _ = _exit_run(TINY, model, n, every=4, extra=1)
    P, L = TINY.prompt_len, TINY.n_layers
    before = _cache(o, TINY, 0, P + n)
    t0, t1 = P + 8, P + 16
    assert o.repass(t0, t1) == 6
    after = _cache(o, TINY, 0, P + n)
    k0 = TINY.readout_layers[0]
    for j in range(L):
        for t in range(P + n):
            kb, vb, sb = before[j][t]
            ka, va, sa = after[j][t]
            inside = t0 <= t < t1 and j >= k0 and sb == 2
            if inside:
                assert sa == 1  # now computed by the layer
                same = np.array_equal(ka, kb) and np.array_equal(va, vb)
                # the first skipped layer's input is the exit residual itself, so
                # its fill was already exact; the layers above it change
                assert same == (j == k0), (j, t)
            else:
                assert sa == sb and np.array_equal(ka, kb) and np.array_equal(va, vb), (j, t)
    # the decode goes on from where it was
    assert o.pos == P + n
    o.decode_step(1, [2.0], oracle.FORCE_FULL)
    with pytest.raises(ValueError):
        o.repass(P, P + n + 5)


# ------------------------------------------------------------- structure
def _trace_step(shape, model, force=oracle.FORCE_FULL, taus=(0.5,)):
    o = oracle.Oracle(shape, model)
    tok = o.prefill(synth.prompt(shape))
    s = o.decode_step(tok, list(taus), force, trace=True)
    return o, tok, s


def test_residual_stream_passes_through_zeroed_layers():
    """With every projection zero, each layer adds nothing: the residual at the
    top is the input token's embedding row, and the logits are the
    unembedding of its RMSNorm."""
    shape = micro()
    model = synth.make_model(shape)
    for lw in model["layers"]:
        for key in ("wq", "wk", "wv", "wo", "wg", "wu", "wd"):
            lw[key] = zeros_like_bits(lw[key])
    o, tok, s = _trace_step(shape, model)
    E = synth.bf16_to_f32(model["embed"])
    h = s["capture"]["h_final"]
    assert np.array_equal(h, E[tok])
    g = synth.bf16_to_f32(model["final_norm"]).astype(np.float64)
    z = E[tok] / np.sqrt(np.mean(E[tok].astype(np.float64) ** 2) + shape.rms_eps) * g
    U = synth.bf16_to_f32(model["lm_head"]).astype(np.float64)
    np.testing.assert_allclose(s["capture"]["final_logits"], U @ z, rtol=1e-5, atol=1e-5)


def test_projection_orientations_and_wiring():
    shape = micro()
    d, A, KH, D, F = shape.d_model, shape.n_heads, shape.n_kv_heads, shape.head_dim, shape.ffn_dim
    model = synth.make_model(shape)
    lw = model["layers"][0]
    lw["wo"] = one_hot_matrix(d, A * D, 5, 17)       # h_mid - h_in = o[17] at row 5
    lw["wd"] = one_hot_matrix(d, F, 9, 40)           # h_out - h_mid = a[40] at row 9
    o, tok, s = _trace_step(shape, model)
    tr = s["capture"]["layer_trace"]
    f = lambda name: o.trace_field(tr, 0, name).astype(np.float64)
    E = synth.bf16_to_f32(model["embed"])
    assert np.array_equal(f("h_in"), E[tok])
    d_attn = f("h_mid") - f("h_in")
    assert d_attn[5] == pytest.approx(f("o")[17], abs=1e-6) and np.count_nonzero(np.delete(d_attn, 5)) == 0
    d_ffn = f("h_out") - f("h_mid")
    assert d_ffn[9] == pytest.approx(f("a")[40], abs=1e-6) and np.count_nonzero(np.delete(d_ffn, 9)) == 0
    # gate and up use W_g and W_u respectively; a = bf16(SiLU(gate) * up)
    u = o.trace_field(tr, 0, "u_mlp")
    np.testing.assert_array_equal(o.trace_field(tr, 0, "gate"), oracle.matvec(lw["wg"], u))
    np.testing.assert_array_equal(o.trace_field(tr, 0, "up"), oracle.matvec(lw["wu"], u))
    g, up = f("gate"), f("up")
    np.testing.assert_array_equal(f("a"), (oracle.silu(g) * up).astype(np.float32))
    # q is W_q u rotated at the step's position; k and v are stored as bf16
    t = o.pos - 1
    ua = o.trace_field(tr, 0, "u_attn")
    q_raw = oracle.matvec(lw["wq"], ua)
    q_rot = np.concatenate([oracle.rope(q_raw[h * D:(h + 1) * D], t, shape.rope_base) for h in range(A)])
    np.testing.assert_array_equal(o.trace_field(tr, 0, "q"), q_rot)
    k_raw = oracle.matvec(lw["wk"], ua)
    k_rot = np.concatenate([oracle.rope(k_raw[g_ * D:(g_ + 1) * D], t, shape.rope_base) for g_ in range(KH)])
    kc, vc, src = o.kv(0, t)
    np.testing.assert_array_equal(kc, bf16_round(k_rot))
    np.testing.assert_array_equal(vc, bf16_round(oracle.matvec(lw["wv"], ua)))


def test_grouped_query_attention_uses_head_div_group():
    """Query head h reads key-value head h div (A/K)."""
    shape = micro()
    A, KH, D = shape.n_heads, shape.n_kv_heads, shape.head_dim
    group = A // KH
    for dead in range(KH):
        model = synth.make_model(shape)
        wv = synth.bf16_to_f32(model["layers"][1]["wv"]).copy()
        wv[dead * D:(dead + 1) * D] = 0
        model["layers"][1]["wv"] = to_bf16_bits(wv)
        o, tok, s = _trace_step(shape, model)
        ov = o.trace_field(s["capture"]["layer_trace"], 1, "o").reshape(A, D)
        for h in range(A):
            assert (np.count_nonzero(ov[h]) == 0) == (h // group == dead)


def test_attention_output_is_softmax_over_cached_positions():
    shape = micro()
    A, KH, D = shape.n_heads, shape.n_kv_heads, shape.head_dim
    model = synth.make_model(shape)
    o, tok, s = _trace_step(shape, model)
    tr = s["capture"]["layer_trace"]
    t = o.pos - 1
    for j in range(shape.n_layers):
        q = o.trace_field(tr, j, "q").reshape(A, D).astype(np.float64)
        Ks = np.stack([o.kv(j, p)[0] for p in range(t + 1)]).reshape(t + 1, KH, D).astype(np.float64)
        Vs = np.stack([o.kv(j, p)[1] for p in range(t + 1)]).reshape(t + 1, KH, D).astype(np.float64)
        got = o.trace_field(tr, j, "o").reshape(A, D)
        for h in range(A):
            g = h // (A // KH)
            p = scipy.special.softmax(Ks[:, g] @ q[h] / math.sqrt(D))
            np.testing.assert_allclose(got[h], p @ Vs[:, g], rtol=1e-5, atol=1e-6)


def test_readout_is_affine_then_final_norm_then_unembedding():
    """Section 2 / Appendix B: y = W_r h + b_r, then the model's own final norm
    and unembedding.  W_r = I + e_i e_j^T checks its orientation."""
    shape = micro()
    d = shape.d_model
    model = synth.make_model(shape)
    W = np.eye(d, dtype=np.float32)
    W[3, 20] = 1.0
    b = np.random.default_rng(3).standard_normal(d).astype(np.float32) * 0.1
    model["readouts"] = [(2, to_bf16_bits(W), to_bf16_bits(b))]
    o = oracle.Oracle(shape, model)
    tok = o.prefill(synth.prompt(shape))
    s = o.decode_step(tok, [1.01], capture=True)
    h = s["capture"]["h_readout"][0].astype(np.float64)
    expect = h + bf16_round(b)
    expect[3] += h[20]
    np.testing.assert_allclose(s["capture"]["y_readout"][0], expect, rtol=1e-6, atol=1e-7)
    y = s["capture"]["y_readout"][0]
    z = oracle.rmsnorm(y, model["final_norm"], shape.rms_eps)
    np.testing.assert_array_equal(s["capture"]["readout_logits"][0], oracle.matvec(model["lm_head"], z))


def test_prefill_equals_forced_full_decode():
    shape = micro()
    model = synth.make_model(shape)
    ids = synth.prompt(shape, shape.prompt_len + 1)
    a = oracle.Oracle(shape, model)
    a.prefill(ids[:-1])
    sa = a.decode_step(int(ids[-1]), [0.5], oracle.FORCE_FULL)
    b = oracle.Oracle(shape, model)
    fb = b.prefill(ids)
    assert sa["token"] == fb
    for j in range(shape.n_layers):
        for t in range(len(ids)):
            ka, va, _ = a.kv(j, t)
            kb, vb, _ = b.kv(j, t)
            assert np.array_equal(ka, kb) and np.array_equal(va, vb)


def _prefill_both_ways(shape, model, parts):
    """Prefill the prompt pieces `parts` (consecutive id arrays) with the
    prefill's matrix products as BLAS calls and position by position."""
    out = []
    n = sum(len(p) for p in parts)
    for gemm in (True, False):
        o = oracle.Oracle(shape, model, max_ctx=n + 2, gemm=gemm)
        toks = [o.prefill(p, capture=True) for p in parts]
        out.append((o, toks))
    return out


@pytest.mark.parametrize("kw,lens", [({}, (100,)), ({"qkv_bias": True}, (7, 600)), ({"n_kv_heads": 1}, (64, 65))])
def test_prefill_matrix_product_form_matches_position_by_position(kw, lens):
    """Long prompts run layer by layer with each projection of a block of
    positions as one BLAS product, and each head's scores and weighted values
    as two more (the block attending to the cache of its layer).  Same steps,
    same float roundings: the cache, the final residual and the logits agree
    with the position-by-position prefill (the products' double sums may
    round differently in the last bit of a float, so a few cache values may
    sit one bf16 step apart).  Covers two blocks of 512 positions, a start
    past position 0 and a prompt that stays position by position (7)."""
    shape = micro(prompt_len=sum(lens), **kw)
    model = synth.make_model(shape)
    ids = synth.prompt(shape, sum(lens))
    parts, at = [], 0
    for n in lens:
        parts.append(ids[at:at + n])
        at += n
    (a, ta), (b, tb) = _prefill_both_ways(shape, model, parts)
    for (xa, ca), (xb, cb) in zip(ta, tb):
        assert xa == xb
        np.testing.assert_allclose(ca["h_final"], cb["h_final"], rtol=1e-5, atol=1e-6)
        np.testing.assert_allclose(ca["final_logits"], cb["final_logits"], rtol=1e-5, atol=1e-5)
    n_diff = n_all = 0
    for j in range(shape.n_layers):
        for t in range(len(ids)):
            ka, va, sa = a.kv(j, t)
            kb, vb, sb = b.kv(j, t)
            assert sa == sb == 1
            for u, v in ((ka, kb), (va, vb)):
                n_diff += int(np.sum(u != v))
                n_all += u.size
                np.testing.assert_allclose(u, v, rtol=2.0 ** -7, atol=1e-6)
    assert n_diff <= n_all // 1000


def test_truncate_then_decode_equals_a_fresh_run():
    """Forgetting the decoded positions and decoding again (another tau, so
    other exits and fills) gives, bit for bit, what a fresh oracle gives."""
    shape = micro()
    model = synth.make_model(shape)
    ids = synth.prompt(shape)
    P, n = len(ids), shape.new_tokens
    a = oracle.Oracle(shape, model)
    first = a.prefill(ids)
    tok = first
    for _ in range(n):
        tok = a.decode_step(tok, [0.0])["token"]
    a.truncate(P)
    assert a.pos == P and a.stats()["steps"] == 0
    b = oracle.Oracle(shape, model)
    assert b.prefill(ids) == first
    ta = tb = first
    for _ in range(n):
        ra, rb = a.decode_step(ta, [0.4]), b.decode_step(tb, [0.4])
        assert ra == rb
        ta, tb = ra["token"], rb["token"]
    assert a.stats() == b.stats()
    for j in range(shape.n_layers):
        for t in range(shape.max_ctx):
            ka, va, sa = a.kv(j, t)
            kb, vb, sb = b.kv(j, t)
            assert sa == sb and np.array_equal(ka, kb) and np.array_equal(va, vb)


def test_qkv_bias_and_tied_head_options():
    shape = micro(qkv_bias=True, tied_embedding=True)
    model = synth.make_model(shape)
    assert model["lm_head"] is None and "bq" in model["layers"][0]
    o, tok, s = _trace_step(shape, model)
    tr = s["capture"]["layer_trace"]
    lw = model["layers"][0]
    ua = o.trace_field(tr, 0, "u_attn")
    t = o.pos - 1
    v_expect = bf16_round(oracle.matvec(lw["wv"], ua) + synth.bf16_to_f32(lw["bv"]))
    np.testing.assert_allclose(o.kv(0, t)[1], v_expect, rtol=1e-2, atol=1e-6)
    # tied: logits use the embedding matrix
    z = oracle.rmsnorm(s["capture"]["h_final"], model["final_norm"], shape.rms_eps)
    np.testing.assert_array_equal(s["capture"]["final_logits"], oracle.matvec(model["embed"], z))


def test_errors_and_determinism():
    shape = micro()
    model = synth.make_model(shape)
    o = oracle.Oracle(shape, model)
    tok = o.prefill(synth.prompt(shape))
    with pytest.raises(ValueError):
        o.decode_step(-1, [0.5])
    with pytest.raises(ValueError):
        o.decode_step(shape.vocab, [0.5])
    for _ in range(shape.new_tokens):
        tok = o.decode_step(tok, [0.5])["token"]
    with pytest.raises(ValueError):
        o.decode_step(tok, [0.5])  # past max_ctx
    _, f1, a = _run(shape, model, [0.4])
    _, f2, b = _run(shape, model, [0.4])
    assert [x["confidence"] for x in a] == [x["confidence"] for x in b]


def _forced_run(shape, model, n, force_of, lazy):
    """Decode n steps with the force values force_of(i); returns (oracle,
    step results)."""
    o = oracle.Oracle(shape, model, max_ctx=shape.prompt_len + n + 1)
    o.set_lazy_fill(lazy)
    tok = o.prefill(synth.prompt(shape))
    taus = [2.0] * len(shape.readout_layers)
    out = []
    for i in range(n):
        s = o.decode_step(tok, taus, force_of(i))
        out.append(s)
        tok = s["token"]
    return o, out


def _same_cache(a, b, shape, t_end):
    for j in range(shape.n_layers):
        for t in range(t_end):
            ka, va, sa = a.kv(j, t)
            kb, vb, sb = b.kv(j, t)
            assert sa == sb and np.array_equal(ka, kb) and np.array_equal(va, vb), (j, t)


def _every4_full(i):
    return oracle.FORCE_FULL if i % 4 == 3 else oracle.FORCE_EXIT_AT(0)


def test_lazy_fill_matches_the_eager_fill():
    """Section 4 step five's fill deferred to the first step that runs the
    layer: no token or confidence changes (an exit step reads only layers
    below its exit), and once flushed the cache is the eager one bit for
    bit (the same projection of the same exit residual)."""
    model = synth.make_model(TINY)
    n = 22
    eager, a = _forced_run(TINY, model, n, _every4_full, False)
    lazy, b = _forced_run(TINY, model, n, _every4_full, True)
    for sa, sb in zip(a, b):
        assert sa["token"] == sb["token"] and sa["exited"] == sb["exited"]
        assert np.array_equal(sa["confidence"], sb["confidence"])
    lazy.flush_fills()
    _same_cache(eager, lazy, TINY, TINY.prompt_len + n)


def test_lazy_fill_waits_for_a_step_that_runs_the_layer():
    model = synth.make_model(TINY)
    P, L, k = TINY.prompt_len, TINY.n_layers, TINY.readout_layers[0]
    eager, _ = _forced_run(TINY, model, 6, _every4_full, False)
    lazy, _ = _forced_run(TINY, model, 6, _every4_full, True)
    # steps 0-2 exited and step 3 ran at full depth: their fills are done
    for t in range(P, P + 3):
        for j in range(k, L):
            assert lazy.kv(j, t)[2] == 2
    _same_cache(eager, lazy, TINY, P + 4)
    # steps 4 and 5 exited after the last full step: still empty above k
    for t in (P + 4, P + 5):
        for j in range(L):
            kl, vl, sl = lazy.kv(j, t)
            if j < k:
                assert sl == 1
            else:
                assert sl == 0 and not kl.any() and not vl.any()
                assert eager.kv(j, t)[2] == 2


def test_lazy_fill_with_readouts_at_several_depths():
    """An exit deeper than a pending one fills that one's entries only in
    the layers it runs; the rest wait for a full step."""
    shape = TINY.replace(readout_layers=(1, 2, 3))
    model = synth.make_model(shape)
    P = shape.prompt_len
    forces = [oracle.FORCE_EXIT_AT(0), oracle.FORCE_EXIT_AT(2), oracle.FORCE_FULL]
    lazy, _ = _forced_run(shape, model, 2, lambda i: forces[i], True)
    assert [lazy.kv(j, P)[2] for j in range(4)] == [1, 2, 2, 0]
    assert [lazy.kv(j, P + 1)[2] for j in range(4)] == [1, 1, 1, 0]
    eager, _ = _forced_run(shape, model, 3, lambda i: forces[i], False)
    lazy, _ = _forced_run(shape, model, 3, lambda i: forces[i], True)
    _same_cache(eager, lazy, shape, P + 3)


def test_lazy_fill_and_the_repass():
    """A re-pass over positions whose fills are still deferred computes the
    same cache as a re-pass after eager fills."""
    model = synth.make_model(TINY)
    P, n = TINY.prompt_len, 14
    eager, _ = _forced_run(TINY, model, n, _every4_full, False)
    lazy, _ = _forced_run(TINY, model, n, _every4_full, True)
    # the last position first: its attention reads the one before it, whose
    # fills are still deferred in the lazy run
    assert eager.repass(P + n - 1, P + n) == lazy.repass(P + n - 1, P + n) == 1
    _same_cache(eager, lazy, TINY, P + n)
    exits = sum(1 for i in range(n - 1) if i % 4 != 3)
    assert eager.repass(P, P + n) == lazy.repass(P, P + n) == exits
    _same_cache(eager, lazy, TINY, P + n)


def test_turning_the_lazy_fill_off_fills_what_is_pending():
    model = synth.make_model(TINY)
    P, n = TINY.prompt_len, 6
    eager, _ = _forced_run(TINY, model, n, _every4_full, False)
    lazy, _ = _forced_run(TINY, model, n, _every4_full, True)
    lazy.set_lazy_fill(False)
    _same_cache(eager, lazy, TINY, P + n)
