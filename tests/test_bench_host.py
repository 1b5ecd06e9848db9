"""Host-side logic of bench.py (no GPU): the replica timing reduction over
ranks (world size 2, gloo), the tau quantile, launch and byte accounting."""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp

import bench
import synth
from paper_2609_14144_gb300 import bytes_model as bm


def _free_port() -> int:
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    r, w, _ = bench.dist_setup()
    assert (r, w) == (rank, world)
    bench.barrier(w)
    # each replica reports its own elapsed time; the job takes the slowest
    out[rank] = bench.max_over_ranks(1.0 + rank * 0.5, w)
    import torch.distributed as dist
    dist.barrier()
    dist.destroy_process_group()


def test_replica_timing_takes_the_slowest_rank():
    world = 2
    out = mp.Manager().dict()
    mp.spawn(_rank_main, args=(world, _free_port(), out), nprocs=world, join=True)
    assert dict(out) == {0: 1.5, 1: 1.5}


def test_tau_for_rate_hits_the_target_fraction():
    rng = np.random.default_rng(0)
    p = rng.random(2047).astype(np.float32)
    for r in (0.08, 0.5, 0.96):
        tau = bench.tau_for_rate(p, r)
        assert abs(np.mean(p > np.float32(tau)) - r) <= 1.0 / len(p) + 1e-9
    assert bench.tau_for_rate(p, 0.0) > 1.0 and bench.tau_for_rate(p, 1.0) == 0.0
    assert np.mean(p > np.float32(bench.tau_for_rate(p, 1.0))) == 1.0


def test_launch_and_byte_accounting_agree_with_the_cost_model():
    sh = synth.CONFIGS["1.5b"]
    L, k = sh.n_layers, sh.readout_layers[0]
    # full step: 5 kernels per layer, readout + vocabulary pass, LM head, step end
    assert bench.step_launches(L, [k], -1) == 5 * L + 2 + 1 + 1
    # exit step: layers up to k, readout + vocabulary pass, KV fill, step end
    assert bench.step_launches(L, [k], 0) == 5 * k + 2 + 1 + 1
    dims = bm.Dims.of(sh)
    kb = bench.kernel_bytes(dims, 700, k)
    per_token_full = (L * (kb["qkv"] + kb["oproj"] + kb["gateup"] + kb["down"] + kb["attention"])
                      + kb["readout"] + 2 * kb["vocab"])
    model_full = bm.step_bytes(dims, 700, [k], None)
    assert per_token_full == pytest.approx(model_full, rel=2e-3)
    lt = bench.kernel_launches_per_token(L, k, 0.5)
    assert lt["gateup"] == k + 0.5 * (L - k) and lt["vocab"] == 1.5 and lt["kvfill"] == 0.5
    # persistent layer kernel: one launch per run of layers between readouts
    assert bench.step_launches(L, [k], -1, True) == 2 + 2 + 1 + 1
    assert bench.step_launches(L, [k], 0, True) == 1 + 2 + 1 + 1
    assert bench.step_launches(L, [7, 14, 21], 1, True) == 2 + 4 + 1 + 1
    assert bench.step_launches(L, [L], -1, True) == 1 + 2 + 1 + 1
    lp = bench.kernel_launches_per_token(L, k, 0.5, True)
    assert lp["qkv"] == 0 and lp["layers"] == 1 + 0.5 * (L - k) / k
    per_token_pers = kb["layers"] * L / k + kb["readout"] + 2 * kb["vocab"]
    assert per_token_pers == pytest.approx(model_full, rel=2e-3)


def test_timed_calls_cover_exactly_the_workload_tokens():
    for n, k in ((512, 20), (512, 5), (1024, 7), (256, 256), (256, 3)):
        sizes = bench.chunk_sizes(n, k)
        assert len(sizes) == k and sum(sizes) == n and max(sizes) - min(sizes) <= 1


def test_thresholds_for_an_overall_exit_rate_over_three_readouts():
    rng = np.random.default_rng(1)
    p = rng.random((2047, 3)).astype(np.float32)
    for r in (0.3, 0.5, 0.8):
        taus = bench.taus_for_overall_rate(p, r)
        overall = np.mean(np.any(p > np.asarray(taus, np.float32)[None, :], axis=1))
        assert abs(overall - r) < 0.01
