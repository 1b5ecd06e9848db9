"""Cost model pins: Table C1 of the paper and the per-step byte counts."""
import json
import os

import pytest

from paper_2609_14144_gb300 import bytes_model as bm
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "table_c1.json")


def _rows():
    with open(GOLDEN) as f:
        return json.load(f)["rows"]


@pytest.mark.parametrize("row", _rows(), ids=lambda r: r["model"])
def test_table_c1_confidence_test_cost(row):
    # Appendix C, Table C1: test cost (H*H + H*V) over one layer's MACs, one decimal.
    le = bm.test_cost_layer_equivalents(row["H"], row["A"], row["K"], row["D"], row["F"], row["V"])
    assert round(le, 1) == pytest.approx(row["test_le"], abs=1e-9)
    share = bm.test_share_of_stack(row["H"], row["A"], row["K"], row["D"], row["F"], row["V"], row["L"])
    assert share == pytest.approx(row["share"], abs=0.006)


def test_7b_unembedding_parameter_count():
    # Appendix C: the 7B unembedding holds about 545 million parameters.
    with open(GOLDEN) as f:
        g = json.load(f)
    row = [r for r in g["rows"] if r["model"] == "Qwen2.5-7B"][0]
    assert row["H"] * row["V"] == pytest.approx(g["unembedding_params_7b"], rel=0.002)


def test_step_bytes_structure():
    m = bm.Dims.of(synth.CONFIGS["1.5b"])
    T = 768
    full = bm.step_bytes(m, T, [14], None)
    ex = bm.step_bytes(m, T, [14], 0)
    plain = bm.plain_step_bytes(m, T)
    # full = plain + one readout + one extra unembedding pass
    assert full - plain == bm.readout_bytes(m) + bm.unembed_bytes(m)
    # the exit step skips 14 layers and adds 14 key/value fills
    assert full - ex == (14 * (bm.layer_weight_bytes(m) + bm.kv_read_bytes(m, T))
                         + bm.unembed_bytes(m) + 2 * m.d - 14 * bm.fill_bytes(m))
    # order of magnitude of the 1.5B numbers (MB per token)
    assert 3.5e9 < full < 3.7e9 and 1.7e9 < ex < 1.9e9 and 3.0e9 < plain < 3.2e9
    # break-even exit rate against the plain model is about a quarter at 1.5B
    r_star = (full - plain) / (full - ex)
    assert 0.2 < r_star < 0.35


def test_mean_bytes_linear_in_exit_rate():
    m = bm.Dims.of(synth.CONFIGS["0.5b"])
    a, b, c = (bm.mean_step_bytes(m, 384, [12], r) for r in (0.0, 0.5, 1.0))
    assert b == pytest.approx((a + c) / 2)
