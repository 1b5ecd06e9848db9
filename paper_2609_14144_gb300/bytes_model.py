"""Cost accounting for the gated decode step.

Two models live here:

* the paper's layer-equivalent cost model (Appendix C): one layer costs
  ``H*A*D + 2*H*K*D + A*D*H + 3*H*F`` multiply-accumulates (four attention
  projections with grouped-query key/value, three gated feed-forward
  matrices); one confidence test costs ``H*H + H*V`` (readout plus
  unembedding);
* the algorithmic HBM bytes a step must move on this implementation: the
  weights of every executed layer, each evaluated readout and its
  unembedding pass, the LM head on full-depth steps, the KV read of every
  executed layer and the KV writes of every layer (computed or filled).
  Skipped layers' weights are not counted: avoiding them is the method.
"""
from __future__ import annotations

import dataclasses


@dataclasses.dataclass(frozen=True)
class Dims:
    L: int   # layers
    d: int   # width (H in Appendix C)
    A: int   # query heads
    K: int   # key-value heads
    D: int   # head dim
    F: int   # feed-forward width
    V: int   # vocabulary

    @classmethod
    def of(cls, shape) -> "Dims":
        return cls(shape.n_layers, shape.d_model, shape.n_heads, shape.n_kv_heads, shape.head_dim,
                   shape.ffn_dim, shape.vocab)


# ------------------------------------------------------------ Appendix C
def layer_macs(H: int, A: int, K: int, D: int, F: int) -> int:
    """Multiply-accumulates of one layer: attention projections + gated FFN."""
    return H * A * D + 2 * H * K * D + A * D * H + 3 * H * F


def test_macs(H: int, V: int) -> int:
    """Multiply-accumulates of one confidence test: readout + unembedding."""
    return H * H + H * V


def test_cost_layer_equivalents(H: int, A: int, K: int, D: int, F: int, V: int) -> float:
    return test_macs(H, V) / layer_macs(H, A, K, D, F)


def test_share_of_stack(H: int, A: int, K: int, D: int, F: int, V: int, L: int) -> float:
    return test_cost_layer_equivalents(H, A, K, D, F, V) / L


# ------------------------------------------------------------ HBM bytes
BF16 = 2


def layer_weight_bytes(m: Dims) -> int:
    """bf16 bytes of one layer: Wq, Wk, Wv, Wo, Wg, Wu, Wd and two norm gains."""
    return BF16 * (m.d * m.A * m.D + 2 * m.d * m.K * m.D + m.A * m.D * m.d + 3 * m.d * m.F + 2 * m.d)


def unembed_bytes(m: Dims) -> int:
    return BF16 * m.V * m.d


def readout_bytes(m: Dims) -> int:
    """W_r (d x d), offset b_r (d) and the final-norm gain (d)."""
    return BF16 * (m.d * m.d + 2 * m.d)


def kv_read_bytes(m: Dims, T: int) -> int:
    """K and V of T positions, one layer."""
    return BF16 * 2 * m.K * m.D * T


def kv_write_bytes(m: Dims) -> int:
    return BF16 * 2 * m.K * m.D


def fill_bytes(m: Dims) -> int:
    """Wk, Wv and the input-norm gain of one skipped layer."""
    return BF16 * (2 * m.d * m.K * m.D + m.d)


def embed_row_bytes(m: Dims) -> int:
    return BF16 * m.d


def step_bytes(m: Dims, T: int, readout_layers, exit_readout: int | None) -> int:
    """Algorithmic bytes of one decode step attending over T positions.

    ``exit_readout`` is the index of the readout that emitted the token, or
    None for a full-depth step (every readout evaluated, then the LM head).
    """
    layers = list(readout_layers)
    per_layer = layer_weight_bytes(m) + kv_read_bytes(m, T) + kv_write_bytes(m)
    if exit_readout is None:
        n_eval = len(layers)
        return (embed_row_bytes(m) + m.L * per_layer + n_eval * (readout_bytes(m) + unembed_bytes(m))
                + unembed_bytes(m) + BF16 * m.d)
    e = layers[exit_readout]
    n_eval = exit_readout + 1
    return (embed_row_bytes(m) + e * per_layer + n_eval * (readout_bytes(m) + unembed_bytes(m))
            + (m.L - e) * (fill_bytes(m) + kv_write_bytes(m)))


def plain_step_bytes(m: Dims, T: int) -> int:
    """Unmodified model: all layers and the LM head, no readout."""
    return step_bytes(m, T, [], None)


def mean_step_bytes(m: Dims, T: int, readout_layers, exit_rate: float) -> float:
    """Single-readout expectation: (1 - r) * full + r * exit."""
    full = step_bytes(m, T, readout_layers, None)
    ex = step_bytes(m, T, readout_layers, 0)
    return (1.0 - exit_rate) * full + exit_rate * ex
