"""Shared helpers for the test suite: small model shapes and weight edits."""
from __future__ import annotations

import numpy as np
import torch

import synth


def micro(**kw) -> synth.ModelShape:
    """A few-layer decoder small enough for brute-force checks."""
    base = dict(name="micro", n_layers=4, d_model=64, n_heads=4, n_kv_heads=2, head_dim=16, ffn_dim=96,
                vocab=300, readout_layers=(2,), seed=7, prompt_len=8, new_tokens=8)
    base.update(kw)
    return synth.ModelShape(**base)


def to_bf16_bits(a) -> np.ndarray:
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16).copy()


def bf16_round(a) -> np.ndarray:
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16).float().numpy()


def bf16_bits_to_f32(a) -> np.ndarray:
    return (np.ascontiguousarray(a, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def damped_after_readout(shape, model: dict, alpha: float) -> dict:
    """The model with the output and down projections of every layer from the
    first readout on scaled by alpha: at alpha = 0 the final residual equals
    the readout layer's, so the readout's answers mostly fall inside the full
    model's nucleus and calibration sees both outcomes."""
    m = dict(model)
    m["layers"] = [dict(l) for l in model["layers"]]
    for j in range(min(shape.readout_layers), shape.n_layers):
        for k in ("wo", "wd"):
            m["layers"][j][k] = to_bf16_bits(bf16_bits_to_f32(model["layers"][j][k]) * alpha)
    return m


def zeros_like_bits(a) -> np.ndarray:
    return np.zeros_like(np.asarray(a, dtype=np.uint16))


def one_hot_matrix(rows: int, cols: int, i: int, j: int, value: float = 1.0) -> np.ndarray:
    m = np.zeros((rows, cols), np.float32)
    m[i, j] = value
    return to_bf16_bits(m)


def identity_bits(n: int) -> np.ndarray:
    return to_bf16_bits(np.eye(n, dtype=np.float32))


# ---------------------------------------------------------------- GPU parity harness
EXCLUDE_EPS = 1e-3    # exclusion band on |p - tau| and on the top-2 probability gap
# |p_gpu - p_oracle| on every evaluated readout.  The comparison rule bounds
# tokens, exit flags, hidden states and logits, not p itself; this bound is a
# sanity check at the size of the drift the bf16 cache allows between two
# correct implementations (an fp32 and an fp64 forward of the 1.5B shape
# differ by up to 1.8e-3 in p at the readout); the observed error is
# reported (EE_PARITY_LOG).
P_TOL = 5e-3
REL_TOL = 1e-2        # max|diff| / max|ref| on hidden states, logits and KV vectors


def parity_log(name: str, **fields):
    """Append one JSON line of parity diagnostics to $EE_PARITY_LOG, if set."""
    import json
    import os
    path = os.environ.get("EE_PARITY_LOG")
    if path:
        with open(path, "a") as f:
            f.write(json.dumps({"test": name, **fields}) + "\n")


def rel_err(a, b) -> float:
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    den = np.max(np.abs(b))
    return float(np.max(np.abs(a - b)) / den) if den > 0 else float(np.max(np.abs(a)))


def is_excluded(o: dict, taus) -> bool:
    """A step whose decision or token sits within the band where rounding
    order may flip it: |p - tau| or a top-2 gap below EXCLUDE_EPS."""
    for r in range(o["n_evaluated"]):
        if abs(o["confidence"][r] - taus[r]) < EXCLUDE_EPS or o["gap"][r] < EXCLUDE_EPS:
            return True
    return (not o["exited"]) and o["full_gap"] < EXCLUDE_EPS


NUC_EPS = 1e-3   # exclusion band on |mass - p_nuc|
MASS_TOL = 2e-3  # |mass_gpu - mass_oracle| outside the ambiguous tokens


def nucleus_ambiguity(final_logits, x: int, p_nuc: float, mass: float):
    """(excluded, bound) for a nucleus check of token x.  Tokens whose logit
    lies within rounding distance of l_x (1e-3 of the largest logit) may fall
    on either side of it; bound is their total probability, by which the
    GPU's mass may differ.  The step is excluded from the bit-exact
    membership check when the oracle's mass lies within NUC_EPS + bound of
    the nucleus share."""
    l = np.asarray(final_logits, np.float64)
    p = np.exp(l - l.max())
    p /= p.sum()
    delta = 1e-3 * max(1.0, float(np.abs(l).max()))
    near = np.abs(l - l[x]) < delta
    near[x] = False
    bound = float(p[near].sum())
    return abs(mass - p_nuc) < NUC_EPS + bound, bound


def forced(o: dict) -> int:
    from paper_2609_14144_gb300 import FORCE_EXIT_AT, FORCE_FULL
    return FORCE_EXIT_AT(o["exit_readout"]) if o["exited"] else FORCE_FULL


def teacher_forced(shape, model, n: int, taus, *, prompt=None, capture: bool = True, graphs: bool = True,
                   pdl: bool = True, persistent: bool = True, page_perm=None, page_size: int = 64,
                   conf_kind: int = 0, nucleus_permille: int = 0):
    """Run the oracle free and the GPU engine teacher-forced on the oracle's
    input tokens and exit decisions.  Returns (first_o, first_g, records,
    oracle, engine)."""
    import oracle
    from paper_2609_14144_gb300 import (OPT_CONFIDENCE, OPT_DEBUG_LOGITS, OPT_GRAPHS, OPT_NUCLEUS, OPT_PDL,
                                        OPT_PERSISTENT, Engine)

    prompt = synth.prompt(shape) if prompt is None else np.asarray(prompt, np.int32)
    max_ctx = len(prompt) + n
    orc = oracle.Oracle(shape, model, max_ctx=max_ctx)
    orc.set_confidence(conf_kind)
    eng = Engine(shape, model, max_ctx=max_ctx, page_size=page_size)
    eng.set_option(OPT_GRAPHS, graphs)
    eng.set_option(OPT_PDL, pdl)
    eng.set_option(OPT_PERSISTENT, 1 if persistent else 0)
    eng.set_option(OPT_CONFIDENCE, conf_kind)
    eng.set_option(OPT_DEBUG_LOGITS, capture)
    if nucleus_permille:
        orc.set_nucleus(nucleus_permille / 1000.0)
        eng.set_option(OPT_NUCLEUS, nucleus_permille)
    if page_perm is not None:
        eng.set_page_table(page_perm)
    first_o = orc.prefill(prompt)
    first_g = eng.prefill(prompt)
    recs, tok = [], first_o
    for _ in range(n):
        o = orc.decode_step(tok, taus, capture=capture)
        g = eng.decode_step(tok, taus, forced(o))
        rec = {"o": o, "g": g, "input": tok}
        if capture:
            rec["g_h"] = [eng.hidden_at_readout(r) for r in range(o["n_evaluated"])]
            rec["g_y"] = [eng.readout_output(r) for r in range(o["n_evaluated"])]
            rec["g_rl"] = [eng.readout_logits(r) for r in range(o["n_evaluated"])]
            if not o["exited"]:
                rec["g_hL"] = eng.hidden_final()
                rec["g_fl"] = eng.final_logits()
        recs.append(rec)
        tok = o["token"]
    return first_o, first_g, recs, orc, eng


def p_errors(recs) -> np.ndarray:
    """|p_gpu - p_oracle| of every evaluated readout of every step."""
    return np.array([abs(r["g"]["confidence"][k] - r["o"]["confidence"][k]) for r in recs
                     for k in range(r["o"]["n_evaluated"])], np.float64)


def check_records(recs, taus, capture: bool = True) -> int:
    """Assert the parity rules; returns the number of excluded steps."""
    excluded = 0
    for i, rec in enumerate(recs):
        o, g = rec["o"], rec["g"]
        assert g["exited"] == o["exited"] and g["exit_readout"] == o["exit_readout"], i
        assert g["n_evaluated"] == o["n_evaluated"], i
        for r in range(o["n_evaluated"]):
            assert abs(g["confidence"][r] - o["confidence"][r]) <= P_TOL, (i, r, g["confidence"], o["confidence"])
        if capture:
            cap = o["capture"]
            for r in range(o["n_evaluated"]):
                assert rel_err(rec["g_h"][r], cap["h_readout"][r]) <= REL_TOL, (i, r)
                assert rel_err(rec["g_y"][r], cap["y_readout"][r]) <= REL_TOL, (i, r)
                assert rel_err(rec["g_rl"][r], cap["readout_logits"][r]) <= REL_TOL, (i, r)
            if not o["exited"]:
                assert rel_err(rec["g_hL"], cap["h_final"]) <= REL_TOL, i
                assert rel_err(rec["g_fl"], cap["final_logits"]) <= REL_TOL, i
        if is_excluded(o, taus):
            excluded += 1
            continue
        assert g["token"] == o["token"], (i, g["token"], o["token"])
        assert g["gate_pass"] == o["gate_pass"], (i, g["gate_pass"], o["gate_pass"])
        assert g["readout_token"] == o["readout_token"], (i, g["readout_token"], o["readout_token"])
        if not o["exited"]:
            assert g["full_token"] == o["full_token"], i
    return excluded


def oracle_steps(orc, first: int, n: int, taus, capture: bool = True) -> list:
    """The oracle free for n steps from its current position (each emitted
    token fed back); records {"o", "input"}."""
    recs, tok = [], first
    for _ in range(n):
        o = orc.decode_step(tok, taus, capture=capture)
        recs.append({"o": o, "input": tok})
        tok = o["token"]
    return recs


def gpu_replay(eng, oracle_recs, taus, capture: bool = True) -> list:
    """The GPU engine teacher-forced on recorded oracle steps (inputs and exit
    decisions); returns records in check_records' form."""
    out = []
    for r in oracle_recs:
        o = r["o"]
        g = eng.decode_step(r["input"], taus, forced(o))
        rec = {"o": o, "g": g, "input": r["input"]}
        if capture:
            rec["g_h"] = [eng.hidden_at_readout(k) for k in range(o["n_evaluated"])]
            rec["g_y"] = [eng.readout_output(k) for k in range(o["n_evaluated"])]
            rec["g_rl"] = [eng.readout_logits(k) for k in range(o["n_evaluated"])]
            if not o["exited"]:
                rec["g_hL"] = eng.hidden_final()
                rec["g_fl"] = eng.final_logits()
        out.append(rec)
    return out


def check_exit_counts(recs, taus, n_readouts: int):
    """Exit counts per readout (and full steps) agree once the excluded steps
    are removed."""
    keep = [r for r in recs if not is_excluded(r["o"], taus)]
    for k in range(n_readouts):
        assert sum(r["g"]["exit_readout"] == k for r in keep) == sum(r["o"]["exit_readout"] == k for r in keep)
    assert sum(not r["g"]["exited"] for r in keep) == sum(not r["o"]["exited"] for r in keep)


def check_kv(orc, eng, shape, n_pos: int, pairs=None):
    """KV positions: which (layer, pos) were written and how, bit for bit;
    values within REL_TOL per vector.  All (layer, pos < n_pos), or the
    given (layer, pos) pairs."""
    if pairs is None:
        pairs = [(j, t) for j in range(shape.n_layers) for t in range(n_pos)]
    for j, t in pairs:
        ko, vo, so = orc.kv(j, t)
        assert eng.kv_src(j, t) == so, (j, t)
        kg, vg = eng.kv(j, t)
        assert rel_err(kg, ko) <= REL_TOL and rel_err(vg, vo) <= REL_TOL, (j, t)
