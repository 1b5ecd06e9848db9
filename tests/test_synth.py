"""The seeded input generator: deterministic, independent streams, the
stated distributions (no GPU)."""
import numpy as np

import synth


def _splitmix64_sequential(state: int, n: int):
    """Textbook SplitMix64 (Steele et al. 2014): state += gamma; mix(state)."""
    M = (1 << 64) - 1
    out = []
    for _ in range(n):
        state = (state + 0x9E3779B97F4A7C15) & M
        z = state
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & M
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & M
        out.append(z ^ (z >> 31))
    return out


def test_counter_stream_is_splitmix64():
    # stream (seed, sid) starts from state mix(seed ^ sid * C); its outputs are
    # the sequential SplitMix64 outputs from that state
    seed, sid = 11, 0
    key = _splitmix64_sequential((seed ^ 0) - 0x9E3779B97F4A7C15 & ((1 << 64) - 1), 1)[0]
    assert list(synth.u64_stream(seed, sid, 0, 6)) == _splitmix64_sequential(key, 6)
    assert list(synth.u64_stream(seed, sid, 3, 3)) == _splitmix64_sequential(key, 6)[3:]


def test_normal_weights_distribution_and_determinism():
    a = synth.normal_bf16(1, 0x1000, (512, 512))
    b = synth.normal_bf16(1, 0x1000, (512, 512))
    c = synth.normal_bf16(1, 0x1001, (512, 512))
    assert np.array_equal(a, b) and not np.array_equal(a, c)
    x = synth.bf16_to_f32(a).astype(np.float64)
    assert abs(x.mean()) < 2e-4 and abs(x.std() - 0.02) < 2e-4
    # Gaussian tails: about 0.27% beyond 3 sigma
    assert 0.0015 < np.mean(np.abs(x) > 0.06) < 0.004


def test_readout_init_and_tokens():
    W = synth.bf16_to_f32(synth.identity_plus_normal_bf16(2, 0x200, 128)).astype(np.float64)
    assert abs(np.diag(W).mean() - 1.0) < 0.01 and abs((W - np.eye(128)).std() - 0.02) < 0.002
    ids = synth.token_ids(2, 0x300, 100000, 151936)
    assert ids.min() >= 0 and ids.max() < 151936 and abs(ids.mean() - 151935 / 2) < 1500
    s = synth.bernoulli(2, 0x400, 100000, 0.26)
    assert abs(s.mean() - 0.26) < 0.005


def test_config_shapes():
    c = synth.CONFIGS["1.5b"]
    assert (c.n_layers, c.d_model, c.n_heads, c.n_kv_heads, c.head_dim, c.ffn_dim, c.vocab) == \
        (28, 1536, 12, 2, 128, 8960, 151936)
    assert synth.CONFIGS["1.5b-long"].readout_layers == (7, 14, 21)
    m = synth.make_model(synth.CONFIGS["tiny"])
    assert m["layers"][0]["wg"].shape == (688, 256) and m["layers"][0]["wd"].shape == (256, 688)
    assert m["lm_head"].shape == m["embed"].shape
