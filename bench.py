#!/usr/bin/env python3
"""Batch-1 decode throughput of the confidence-gated early-exit path on GB300.

Workload: the 1.5B-shaped synthetic decoder (28 layers, width 1536, 12/2
heads of 128, SwiGLU 8960, vocabulary 151936) with a readout at layer 14,
a 512-token prompt and 512 greedy tokens.  tau is calibrated as the quantile
of the readout's top-1 probability over a seeded 2048-token calibration
stream (teacher-forced at full depth) to hit the target exit rate.

The timed region decodes exactly the workload's 512 greedy tokens after the
prompt, in --steps ee_decode_n calls (one benchmark step = one call: a graph
launch running its share of the gated decode steps with on-device token
feedback).  --warmup calls run first on a sequence of their own; the prompt is
then prefilled again outside the timed region.

The JSON line reports tokens/s at the 50% exit target, the exit-rate sweep
(calibrated tau and imposed exits), the unmodified model (no readout) as the
speedup denominator, the 0.5B, 3B and long-context workloads at their own
calibrated exit rates, the achieved HBM bandwidth of the whole step from the
algorithmic byte count, the dominant kernel's roofline, an end-to-end number
through the host-buffer API, SM clocks during the timed region, and the CPU
oracle's speed on a bounded sample.  ``--impl reference`` times the CPU
oracle alone (the reference arm).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import synth  # noqa: E402
from paper_2609_14144_gb300 import bytes_model as bm  # noqa: E402

METRIC = "decode tokens/sec at batch 1 vs exit rate; achieved HBM GB/s as % of roofline"
UNIT = "tokens/s"
WORKLOAD = "1.5b"
HEADLINE_RATE = 0.5
CALIB_TOKENS = 2048
REPASS_W = 16  # positions in the measured full-depth re-pass
ROWS_MAX = 256  # positions per batch of the multi-position layer pass (EE_OPT_ROWS)
CTL_BYTES = 368  # device control block read back by a host-buffer ee_decode_n


def _peaks() -> dict:
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "source": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "source": "fallback"}


def _log(*a):
    print(*a, file=sys.stderr, flush=True)


# --------------------------------------------------------------------- distributed
def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist

        import torch
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        dist.init_process_group(backend)
    return rank, world, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# --------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi samples every 200 ms while running."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu: int):
        self.gpu = gpu
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                self.proc.wait(5)
            except Exception:
                self.proc.kill()

    def summary(self) -> dict:
        rows = []
        try:
            with open(self.path) as f:
                for line in f:
                    parts = [p.strip() for p in line.split(",")]
                    if len(parts) >= 9:
                        rows.append(parts)
            os.remove(self.path)
        except Exception:
            pass
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


# --------------------------------------------------------------------- helpers
def tau_for_rate(p: np.ndarray, rate: float) -> float:
    """Lowest tau with a fraction `rate` of p strictly above it:
    tau = p_(ceil((1 - rate) N)) in ascending order; rate 0 -> 1.01, 1 -> 0."""
    if rate <= 0.0:
        return 1.01
    if rate >= 1.0:
        return 0.0
    s = np.sort(np.asarray(p, np.float32))
    k = int(math.ceil((1.0 - rate) * len(s)))
    return float(s[max(0, min(len(s) - 1, k - 1))])


def layer_launches(L: int, bounds, persistent: bool) -> int:
    """Launches that run layers [b_i, b_{i+1}) for consecutive bounds: five per
    layer, or one persistent launch per non-empty run."""
    runs = [b - a for a, b in zip(bounds[:-1], bounds[1:])]
    return sum(1 for r in runs if r > 0) if persistent else 5 * sum(runs)


def step_launches(L: int, readout_layers, exit_readout: int, persistent: bool = False) -> int:
    """Kernels one gated decode step launches (graph nodes of libee)."""
    ro = list(readout_layers)
    if exit_readout < 0:
        return layer_launches(L, [0] + ro + [L], persistent) + 2 * len(ro) + 1 + 1
    e = ro[exit_readout]
    return layer_launches(L, [0] + ro[:exit_readout + 1], persistent) + 2 * (exit_readout + 1) + \
        (1 if e < L else 0) + 1


def kernel_bytes(dims: bm.Dims, T: int, k_layer: int) -> dict:
    """Algorithmic HBM bytes of one launch of each decode kernel."""
    d, A, K, D, F, V, L = dims.d, dims.A, dims.K, dims.D, dims.F, dims.V, dims.L
    return {
        "qkv": 2 * ((A + 2 * K) * D * d + d) + 4 * K * D,
        "attention": 4 * K * D * T,
        "oproj": 2 * d * A * D,
        "gateup": 2 * (2 * F * d + d),
        "down": 2 * d * F,
        "readout": 2 * (d * d + d),
        "vocab": 2 * (V * d + d),
        "kvfill": (L - k_layer) * (2 * (2 * K * D * d + d) + 4 * K * D),
        # the persistent kernel over layers 1..k: their weights and KV traffic
        "layers": k_layer * (2 * ((A + 2 * K) * D * d + d) + 4 * K * D + 4 * K * D * T + 2 * d * A * D
                             + 2 * (2 * F * d + d) + 2 * d * F),
    }


def kernel_launches_per_token(L: int, k: int, exit_rate: float, persistent: bool = False) -> dict:
    """Launches of each kernel per token.  With the persistent kernel, the
    upper run of layers counts as (L - k) / k launches of the measured
    layers-1..k launch (same per-layer work)."""
    full = 1.0 - exit_rate
    layers = k + full * (L - k)
    out = {"readout": 1.0, "vocab": 1.0 + full, "kvfill": exit_rate}
    if persistent:
        out.update({"qkv": 0.0, "attention": 0.0, "oproj": 0.0, "gateup": 0.0, "down": 0.0,
                    "layers": 1.0 + full * (L - k) / k})
    else:
        out.update({"qkv": layers, "attention": layers, "oproj": layers, "gateup": layers, "down": layers,
                    "layers": 0.0})
    return out


def ncu_traffic(kernel: str, shape_name: str, attended: int | None = None, dims=None) -> float | None:
    """Per-launch DRAM bytes from a committed ncu summary, if its recorded
    kernel-source hash still matches the current source.  For the layer
    kernel, the capture's cache reads are moved to `attended` positions (the
    weights do not depend on the position)."""
    path = os.path.join(ROOT, "profiles", f"ncu_{kernel}_{shape_name.replace('.', 'p')}.md")
    if not os.path.exists(path):
        return None
    vals = {}
    for line in open(path):
        if ":" in line and line.strip().startswith("- "):
            k, v = line.strip()[2:].split(":", 1)
            vals[k.strip()] = v.strip()
    src_name = vals.get("kernel_source", "ee_kernels.cu")
    src = open(os.path.join(ROOT, "paper_2609_14144_gb300", "csrc", src_name), "rb").read()
    if vals.get("kernel_source_sha256") != hashlib.sha256(src).hexdigest()[:16]:
        return None
    try:
        traffic = float(vals["dram_bytes_per_launch"])
        if attended is not None and dims is not None and "attended_positions" in vals:
            layers = int(vals.get("layers_per_launch", "1"))
            traffic += layers * 4 * dims.K * dims.D * (attended - int(vals["attended_positions"]))
        return traffic
    except Exception:
        return None


def oracle_sample(shape, model, seconds: float, prompt_len: int = 16, rate: float = HEADLINE_RATE,
                  min_steps: int = 4) -> dict:
    """Time the CPU oracle's gated decode on a bounded sample of the workload:
    a short prompt, then steps with exits imposed at `rate` (the same byte
    mix), until `seconds` of decode work."""
    import oracle

    orc = oracle.Oracle(shape, model, max_ctx=prompt_len + 4096)
    ids = synth.prompt(shape, prompt_len)
    tok = orc.prefill(ids)
    sched = synth.exit_schedule(shape, 4096, rate, index=7)
    t0 = time.perf_counter()
    n = 0
    while n < min_steps or (time.perf_counter() - t0) < seconds:
        force = oracle.FORCE_EXIT_AT(0) if sched[n] else oracle.FORCE_FULL
        tok = orc.decode_step(tok, [0.5], force)["token"]
        n += 1
    dt = time.perf_counter() - t0
    cores = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    return {"value": n / dt, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{shape.name}: {prompt_len}-token prompt, {n} gated decode steps with exits imposed "
                      f"at {rate:.0%} (Bernoulli schedule), {dt:.1f} s of CPU work"}


def run_reference(args, rank: int, world: int):
    """Reference arm: the CPU oracle as it stands, on the host cores."""
    if rank != 0:
        return
    shape = synth.CONFIGS[WORKLOAD]
    t0 = time.perf_counter()
    model = synth.make_model(shape)
    _log(f"[reference] model generated in {time.perf_counter() - t0:.1f} s")
    import oracle

    tokens_per_step = 2
    P = shape.prompt_len
    orc = oracle.Oracle(shape, model, max_ctx=P + tokens_per_step * (args.steps + args.warmup))
    tok = orc.prefill(synth.prompt(shape, P))
    sched = synth.exit_schedule(shape, 4096, HEADLINE_RATE, index=7)
    i = 0

    def one_step():
        nonlocal tok, i
        for _ in range(tokens_per_step):
            force = oracle.FORCE_EXIT_AT(0) if sched[i] else oracle.FORCE_FULL
            tok = orc.decode_step(tok, [0.5], force)["token"]
            i += 1

    for _ in range(args.warmup):
        one_step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        one_step()
    dt = time.perf_counter() - t0
    value = args.steps * tokens_per_step / dt
    cores = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    sample = (f"{shape.name}: {P}-token prompt, {tokens_per_step} gated decode steps per benchmark step with exits "
              f"imposed at {HEADLINE_RATE:.0%} (Bernoulli schedule), {args.steps} timed steps")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": dt / args.steps * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": _workload_desc(shape), "exit_rate_target": HEADLINE_RATE,
                       "exits": "imposed Bernoulli(0.5) schedule (same byte mix; no calibration pass)"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def _workload_desc(shape) -> str:
    return (f"{shape.name}-shaped decoder: L{shape.n_layers} d{shape.d_model} A{shape.n_heads}/K{shape.n_kv_heads} "
            f"D{shape.head_dim} F{shape.ffn_dim} V{shape.vocab}, readout at layer {shape.readout_layers[0]}, "
            f"prompt {shape.prompt_len}, {shape.new_tokens} greedy tokens, batch 1")


# --------------------------------------------------------------------- GPU arm
def chunk_sizes(n_new: int, steps: int) -> list:
    """`steps` chunk lengths that add up to n_new tokens (the first n_new mod
    steps one longer)."""
    base, extra = divmod(n_new, steps)
    return [base + (1 if i < extra else 0) for i in range(steps)]


class Runner:
    """Timed decodes of one workload: the prompt is prefilled outside the
    timed region, then the workload's new tokens are decoded in `steps`
    ee_decode_n calls (benchmark steps) that together produce exactly the
    configuration's number of greedy tokens.  Warm-up calls run on a sequence
    of their own, before a reset and a fresh prefill."""

    def __init__(self, eng, shape, world, n_new):
        import torch
        self.torch = torch
        self.eng, self.shape, self.world, self.n_new = eng, shape, world, n_new
        self.dims = bm.Dims.of(shape)

    def _prefill(self, prompt):
        self.eng.reset()
        self.eng.prefill(prompt)

    def run(self, taus, warmup, steps, schedule=None, prompt=None, clocks=None):
        torch, eng = self.torch, self.eng
        from paper_2609_14144_gb300 import DEVICE
        prompt = synth.prompt(self.shape) if prompt is None else prompt
        P, n = len(prompt), self.n_new
        sizes = chunk_sizes(n, steps)
        tok = torch.empty(n, dtype=torch.int32, device=eng.device)
        ex = torch.empty(n, dtype=torch.int32, device=eng.device)
        cf = torch.empty(n, dtype=torch.float32, device=eng.device)
        if warmup:
            self._prefill(prompt)
            at = 0
            for i in range(warmup):
                c = min(sizes[0], n - at)
                if c <= 0:
                    break
                sch = None if schedule is None else schedule[at:at + c]
                eng.decode_n(c, taus, schedule=sch, where=DEVICE, tokens=tok[at:at + c], exit_readout=ex[at:at + c],
                             confidence=cf[at:at + c])
                at += c
            eng.sync()
        self._prefill(prompt)
        barrier(self.world)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        ctx = clocks if clocks is not None else _Null()
        with ctx:
            e0.record(eng.stream)
            at = 0
            for c in sizes:
                sch = None if schedule is None else schedule[at:at + c]
                eng.decode_n(c, taus, schedule=sch, where=DEVICE, tokens=tok[at:at + c], exit_readout=ex[at:at + c],
                             confidence=cf[at:at + c])
                at += c
            e1.record(eng.stream)
            e1.synchronize()
        torch.cuda.synchronize()
        eng.sync()
        ms = e0.elapsed_time(e1)
        ms_max = max_over_ranks(ms, self.world)
        exits = ex.cpu().numpy()
        ro = list(self.shape.readout_layers)
        bytes_total = sum(bm.step_bytes(self.dims, P + i + 1, ro, None if e < 0 else int(e))
                          for i, e in enumerate(exits))
        launches = sum(step_launches(self.shape.n_layers, ro, int(e), self.eng.persistent) for e in exits) + steps
        return {"ms": ms_max, "tokens": n * self.world, "tok_s": n * self.world / (ms_max / 1e3),
                "exit_rate": float(np.mean(exits >= 0)) if len(ro) else 0.0,
                "exits_by_readout": [int(np.sum(exits == k)) for k in range(len(ro))],
                "bytes_per_token": bytes_total / n, "gbs": bytes_total * self.world / (ms_max / 1e3) / 1e9,
                "launches": launches, "tokens_out": tok.cpu().numpy(), "exits": exits,
                "attended": [P + 1, P + n]}

    def run_host(self, taus, warmup, steps, prompt):
        """The same decode through the host-buffer API: every call copies tau
        in and its tokens, exits and confidences (and the control block) back
        and synchronises (end to end)."""
        eng, n = self.eng, self.n_new
        sizes = chunk_sizes(n, steps)
        self._prefill(prompt)
        at = 0
        for _ in range(warmup):
            c = min(sizes[0], n - at)
            if c <= 0:
                break
            eng.decode_n(c, taus)
            at += c
        self._prefill(prompt)
        barrier(self.world)
        t0 = time.perf_counter()
        for c in sizes:
            eng.decode_n(c, taus)
        dt = max_over_ranks(time.perf_counter() - t0, self.world)
        return n * self.world / dt


class _Null:
    def __enter__(self):
        return self

    def __exit__(self, *a):
        return False


def calibrate(eng, shape, n: int = CALIB_TOKENS, p_nuc: float = 0.9, fidelity: float = 0.9):
    """The on-device calibration pass over a seeded stream (teacher-forced at
    full depth, one graph launch): every readout's top-1 probability and
    readout 0's membership in the full model's nucleus, then the threshold
    selection at the fidelity target.  Returns (p [n-1, R], summary)."""
    import torch

    from paper_2609_14144_gb300 import DEVICE, select_tau
    stream = synth.calibration_stream(shape, n)
    eng.reset()
    eng.prefill(stream[:1])
    ids = torch.from_numpy(np.asarray(stream[1:], np.int32)).to(eng.device)
    torch.cuda.synchronize(eng.device)
    t0 = time.perf_counter()
    conf, member, _ = eng.calibrate(ids, p_nuc, where=DEVICE)
    tau = select_tau(conf[:, 0], member, fidelity, stream=eng.stream)
    eng.sync()
    dt = time.perf_counter() - t0
    p = conf.cpu().numpy()
    t = float(tau.item())  # -inf: every position may exit; +inf: no threshold reaches the target
    summary = {"tokens": n - 1, "s": dt, "tok_s": (n - 1) / dt, "nucleus": p_nuc, "fidelity_target": fidelity,
               "acceptable_share": float(member.float().mean().item()),
               "fidelity_tau": t if math.isfinite(t) else ("-inf" if t < 0 else "+inf"),
               "note": "Section 4 step four on synthetic weights: the readout's answers rarely fall in the full "
                       "model's nucleus, so the fidelity threshold admits few or no exits; the timed runs use "
                       "the exit-rate quantile threshold"}
    eng.reset()
    return p, summary


def taus_for_overall_rate(p: np.ndarray, rate: float) -> list:
    """Thresholds for several readouts (shallowest first, first passing one
    exits): every readout at the same per-readout quantile level, chosen by
    bisection so that the share of calibration positions at which some
    readout passes is about `rate`."""
    lo, hi = 0.0, rate
    taus = None
    for _ in range(40):
        mid = 0.5 * (lo + hi)
        taus = [tau_for_rate(p[:, k], mid) for k in range(p.shape[1])]
        overall = float(np.mean(np.any(p > np.asarray(taus, np.float32)[None, :], axis=1)))
        if overall < rate:
            lo = mid
        else:
            hi = mid
    return taus


def kernel_roofline(eng, run, shape, prompt, taus, exit_rate, W_tokens, peak) -> dict:
    """Per-kernel device time (direct launches, CUDA events on the engine's
    stream) after a prefill and W_tokens decoded tokens, and the dominant
    kernel's algorithmic GB/s against the measured copy bandwidth."""
    eng.reset()
    eng.prefill(prompt)
    if W_tokens:
        eng.decode_n(W_tokens, taus)
    kms = eng.profile_kernels(iters=2 * shape.n_layers)
    T_prof = eng.position + 1
    kb = kernel_bytes(run.dims, T_prof, shape.readout_layers[0])
    per_tok = kernel_launches_per_token(shape.n_layers, shape.readout_layers[0], exit_rate, eng.persistent)
    share = {k: kms[k] * per_tok[k] for k in kms}
    dom = max(share, key=share.get)
    ach = kb[dom] / (kms[dom] / 1e3) / 1e9
    return {"bound": "hbm", "kernel": dom, "achieved": ach, "peak": peak["hbm_gbs"], "unit": "GB/s",
            "frac": ach / peak["hbm_gbs"], "peak_source": peak["source"],
            "traffic": ncu_traffic(dom, shape.name, T_prof, run.dims), "bytes_per_launch": kb[dom],
            "ms_per_launch": kms[dom], "attended_positions": T_prof,
            "kernels": {k: {"ms": kms[k], "GBps": kb[k] / (kms[k] / 1e3) / 1e9 if kms[k] > 0 else None,
                            "share": share[k] / sum(share.values())} for k in kms}}


def extra_workload(name: str, args, world: int, local: int, peak: dict) -> dict:
    """Decode throughput of another workload at its calibrated exit rates:
    its own prompt and new-token count, the timed region covering exactly
    those tokens (args.steps calls, one warm-up call), the step's algorithmic
    GB/s and its fraction of the measured copy bandwidth, and the layer
    kernel's roofline."""
    import torch

    from paper_2609_14144_gb300 import Engine

    shape = synth.CONFIGS[name]
    t0 = time.perf_counter()
    model = synth.make_model(shape)
    prompt = synth.prompt(shape)
    eng = Engine(shape, model, max_ctx=max(shape.prompt_len + shape.new_tokens, CALIB_TOKENS), device=local)
    run = Runner(eng, shape, world, shape.new_tokens)
    p_all, _ = calibrate(eng, shape)
    # the prompt itself, batched on the tensor cores (the default): not part of the timed decode
    eng.reset()
    torch.cuda.synchronize(local)
    t0p = time.perf_counter()
    eng.prefill(prompt)
    prefill_ms = (time.perf_counter() - t0p) * 1e3
    if len(shape.readout_layers) > 1:
        plan = [(r, taus_for_overall_rate(p_all, r)) for r in shape.exit_rates]
    else:
        plan = [(r, [tau_for_rate(p_all[:, 0], r)]) for r in shape.exit_rates]
    sweep = []
    for r, taus in plan:
        res = run.run(taus, 1, args.steps, prompt=prompt)
        sweep.append({"target_rate": r, "tau": taus if len(taus) > 1 else taus[0], "exit_rate": res["exit_rate"],
                      "exits_by_readout": res["exits_by_readout"], "tok_s": res["tok_s"], "GBps": res["gbs"],
                      "frac": res["gbs"] / peak["hbm_gbs"], "MB_per_token": res["bytes_per_token"] / 1e6})
        _log(f"[bench] {name} r={r}: rate={res['exit_rate']:.3f} {res['tok_s']:.1f} tok/s {res['gbs']:.0f} GB/s")
    mid = plan[len(plan) // 2]
    roof = kernel_roofline(eng, run, shape, prompt, mid[1], sweep[len(plan) // 2]["exit_rate"],
                           min(64, shape.new_tokens), peak)
    eng.close()
    del eng, model
    return {"workload": _workload_desc(shape), "timed": f"{shape.new_tokens} tokens after the {shape.prompt_len}-"
            f"token prompt in {args.steps} calls", "sweep": sweep, "roofline": roof,
            "prefill_ms": prefill_ms, "s": time.perf_counter() - t0}


def run_ours(args, rank: int, world: int, local: int):
    import torch

    from paper_2609_14144_gb300 import FORCE_EXIT_AT, FORCE_FULL, OPT_LAZY_FILL, OPT_ROWS, Engine

    torch.cuda.set_device(local)
    shape = synth.CONFIGS[WORKLOAD]
    W, K = args.warmup, args.steps
    n_new = shape.new_tokens
    t0 = time.perf_counter()
    model = synth.make_model(shape.replace(seed=shape.seed))
    prompt = synth.token_ids(shape.seed + 1000 * rank, synth.SID_PROMPT, shape.prompt_len, shape.vocab)
    _log(f"[bench] rank {rank}: model generated in {time.perf_counter() - t0:.1f} s")
    max_ctx = max(shape.prompt_len + n_new, CALIB_TOKENS)
    eng = Engine(shape, model, max_ctx=max_ctx, device=local)
    run = Runner(eng, shape, world, n_new)
    peak = _peaks()

    t0 = time.perf_counter()
    p_all, cal = calibrate(eng, shape)
    p_cal = p_all[:, 0]
    _log(f"[bench] calibration ({CALIB_TOKENS} tokens) in {time.perf_counter() - t0:.1f} s "
         f"(on-device pass {cal['s'] * 1e3:.0f} ms); p quantiles "
         f"{np.quantile(p_cal, [0.04, 0.5, 0.92]).round(3).tolist()}; acceptable share "
         f"{cal['acceptable_share']:.3f}, fidelity tau {cal['fidelity_tau']}")
    taus = {r: tau_for_rate(p_cal, r) for r in sorted(set(shape.exit_rates) | {HEADLINE_RATE})}

    # headline: calibrated tau at the 50% target
    tau_h = taus[HEADLINE_RATE]
    run.run([tau_h], 1, K, prompt=prompt)  # build graphs, warm the path
    clocks = ClockSampler(local)
    head = run.run([tau_h], W, K, prompt=prompt, clocks=clocks)
    clk = clocks.summary()
    _log(f"[bench] headline tau={tau_h:.4f}: {head['tok_s']:.1f} tok/s, exit rate {head['exit_rate']:.3f}, "
         f"{head['gbs']:.0f} GB/s, clocks {clk}")

    sweep = []
    if not args.no_sweep:
        for r in sorted(taus):
            res = run.run([taus[r]], 1, K, prompt=prompt)
            sched = np.where(synth.exit_schedule(shape, n_new, r, index=1) == 1, FORCE_EXIT_AT(0),
                             FORCE_FULL).astype(np.int8)
            imp = run.run([0.5], 1, K, schedule=sched, prompt=prompt)
            # the same decode with the deferred fill (the byte count above assumes eager fills)
            eng.set_option(OPT_LAZY_FILL, 1)
            lz = run.run([taus[r]], 1, K, prompt=prompt)
            eng.set_option(OPT_LAZY_FILL, 0)
            sweep.append({"target_rate": r, "tau": taus[r], "exit_rate": res["exit_rate"],
                          "tok_s": res["tok_s"], "GBps": res["gbs"], "frac": res["gbs"] / peak["hbm_gbs"],
                          "MB_per_token": res["bytes_per_token"] / 1e6,
                          "imposed": {"exit_rate": imp["exit_rate"], "tok_s": imp["tok_s"], "GBps": imp["gbs"],
                                      "frac": imp["gbs"] / peak["hbm_gbs"],
                                      "MB_per_token": imp["bytes_per_token"] / 1e6},
                          "deferred_fill": {"exit_rate": lz["exit_rate"], "tok_s": lz["tok_s"],
                                            "speedup": lz["tok_s"] / res["tok_s"]}})
            _log(f"[bench] sweep r={r}: tau={taus[r]:.4f} rate={res['exit_rate']:.3f} {res['tok_s']:.1f} tok/s "
                 f"{res['gbs']:.0f} GB/s | imposed rate={imp['exit_rate']:.3f} {imp['tok_s']:.1f} tok/s | "
                 f"deferred fill {lz['tok_s']:.1f} tok/s")

    # the unmodified model (no readout): the speedup denominator
    plain_line = None
    if not args.no_sweep:
        eng_plain = Engine(shape, model, max_ctx=max_ctx, device=local, readouts=False)
        rp = Runner(eng_plain, shape.replace(readout_layers=()), world, n_new)
        pl = rp.run(None, 1, K, prompt=prompt)
        plain_line = {"tok_s": pl["tok_s"], "GBps": pl["gbs"], "frac": pl["gbs"] / peak["hbm_gbs"],
                      "MB_per_token": pl["bytes_per_token"] / 1e6,
                      "speedup_at_headline": head["tok_s"] / pl["tok_s"]}
        _log(f"[bench] plain model: {pl['tok_s']:.1f} tok/s, {pl['gbs']:.0f} GB/s")
        eng_plain.close()
        del eng_plain

    # Section 11's full-depth re-pass: decode REPASS_W tokens with every
    # step exiting, then time one re-pass of them (ee_repass)
    # (timed for the batched pass and for one position at a time)
    repass = None
    if not args.no_sweep:
        repass = {"positions": REPASS_W}
        for rows in (1, 0, 1):  # the first batched run warms up
            eng.set_option(OPT_ROWS, rows)
            eng.reset()
            eng.prefill(prompt)
            sched = np.full(REPASS_W, FORCE_EXIT_AT(0), np.int8)
            eng.decode_n(REPASS_W, [0.5], schedule=sched)
            p1 = eng.position
            torch.cuda.synchronize(local)
            t0 = time.perf_counter()
            n_rp = eng.repass(p1 - REPASS_W, p1)
            dt = time.perf_counter() - t0
            key = "batched" if rows else "one_position_at_a_time"
            repass[key] = {"repassed": n_rp, "ms": dt * 1e3, "token_times": dt * head["tok_s"]}
        eng.set_option(OPT_ROWS, 1)
        b = repass["batched"]
        _log(f"[bench] re-pass of {b['repassed']} exited positions: {b['ms']:.2f} ms ({b['token_times']:.2f} "
             f"token-times); one position at a time {repass['one_position_at_a_time']['ms']:.2f} ms")

    # the prompt: batches of up to ROWS_MAX positions, and one position at a time
    prefill = None
    if not args.no_sweep:
        P = len(prompt)
        batches = -(-P // ROWS_MAX)
        prefill = {"positions": P, "batch_rows": ROWS_MAX}
        for rows in (1, 1, 0):  # the first batched run warms up
            eng.set_option(OPT_ROWS, rows)
            eng.reset()
            torch.cuda.synchronize(local)
            t0 = time.perf_counter()
            eng.prefill(prompt)
            dt = time.perf_counter() - t0
            key = "batched" if rows else "one_position_at_a_time"
            passes = batches if rows else P
            prefill[key] = {"ms": dt * 1e3, "tok_s": P / dt,
                            "weight_GBps": passes * bm.layer_weight_bytes(run.dims) * shape.n_layers / dt / 1e9}
        eng.set_option(OPT_ROWS, 1)
        _log(f"[bench] prompt of {P}: {prefill['batched']['ms']:.2f} ms batched "
             f"({prefill['batched']['tok_s']:.0f} tok/s), {prefill['one_position_at_a_time']['ms']:.1f} ms "
             f"one position at a time")

    # end to end through the host-buffer API
    e2e = run.run_host([tau_h], W, K, prompt)

    # per-kernel device time (direct launches) and the dominant kernel's roofline
    roofline = kernel_roofline(eng, run, shape, prompt, [tau_h], head["exit_rate"], n_new // 2, peak)
    step_roof = {"achieved": head["gbs"], "peak": peak["hbm_gbs"], "unit": "GB/s",
                 "frac": head["gbs"] / peak["hbm_gbs"], "frac_of_nominal_7900": head["gbs"] / 7900.0,
                 "MB_per_token": head["bytes_per_token"] / 1e6}
    eng.close()
    del eng

    # the other large workloads, each at its calibrated exit rates
    workloads = {}
    if not args.no_sweep and world == 1:
        for name in ("0.5b", "3b", "1.5b-long"):
            workloads[name] = extra_workload(name, args, world, local, peak)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        cpu = oracle_sample(shape, model, seconds=args.cpu_seconds, prompt_len=shape.prompt_len)
        _log(f"[bench] cpu oracle: {cpu['value']:.2f} tok/s on {cpu['cores']} cores")

    ms_per_step = head["ms"] / K
    line = {
        "metric": METRIC, "value": head["tok_s"], "unit": UNIT, "n_gpus": world, "steps": K, "warmup": W,
        "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic",
        "config": {"workload": _workload_desc(shape),
                   "timed": f"the {n_new} greedy tokens after the {shape.prompt_len}-token prompt (attended "
                            f"positions {head['attended'][0]}..{head['attended'][1]}), in {K} ee_decode_n calls of "
                            f"{min(chunk_sizes(n_new, K))}-{max(chunk_sizes(n_new, K))} tokens; warm-up calls on a "
                            f"sequence of their own",
                   "exit_rate_target": HEADLINE_RATE, "tau": tau_h, "exit_rate": head["exit_rate"],
                   "parallelism": f"replicas x{world}",
                   "l2": "inputs larger than L2: every token streams 1.8-3.6 GB of weights",
                   "numerics": "bf16 weights and KV cache, fp32 activations and accumulation (values exchanged "
                               "between CTAs whole fp32; attention scores from three bf16 parts of the query on "
                               "the tensor cores, exact products)"},
        "e2e": {"value": e2e, "unit": UNIT, "h2d_bytes_per_step": 4 * 8,
                "d2h_bytes_per_step": 12 * max(chunk_sizes(n_new, K)) + CTL_BYTES},
        "gpu_launches": head["launches"],
        "roofline": roofline,
        "step_roofline": step_roof,
        "cpu_baseline": cpu,
        "clocks": clk,
        "sweep": sweep,
        "plain_model": plain_line,
        "workloads": workloads,
        "calibration": cal,
        "repass": repass,
        "prefill": prefill,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)


def profile_run(args, local: int):
    """A short decode for ncu captures: 64-token prompt, two 8-token chunks
    with exits imposed at 50%, no calibration.  Prints the launch counts.
    --eager launches every kernel directly (ncu cannot profile single kernel
    nodes of graphs that hold conditional nodes).  The prompt runs one position
    at a time, so the launches before the decode steps are the fixed count
    printed here."""
    import torch

    from paper_2609_14144_gb300 import DEVICE, FORCE_EXIT_AT, FORCE_FULL, OPT_GRAPHS, OPT_ROWS, Engine

    torch.cuda.set_device(local)
    shape = synth.CONFIGS[WORKLOAD]
    model = synth.make_model(shape)
    if args.rows:
        return profile_rows(shape, model, local)
    P, C = 64, 8
    eng = Engine(shape, model, max_ctx=P + 2 * C, device=local)
    if args.eager:
        eng.set_option(OPT_GRAPHS, 0)
    eng.set_option(OPT_ROWS, 0)
    eng.prefill(synth.prompt(shape, P))
    sched = np.where(synth.exit_schedule(shape, 2 * C, 0.5, index=1) == 1, FORCE_EXIT_AT(0), FORCE_FULL)
    sched = sched.astype(np.int8)
    for i in range(2):
        eng.decode_n(C, [0.5], schedule=sched[i * C:(i + 1) * C], where=DEVICE)
    eng.sync()
    L = shape.n_layers
    prefill_launches = 1 + P * (layer_launches(L, [0, L], eng.persistent) + 1) + 2
    decode = sum(step_launches(L, shape.readout_layers, 0 if e else -1, eng.persistent) for e in (sched >= 2)) + 2
    print(json.dumps({"prefill_launches": prefill_launches, "decode_launches": decode, "tokens": 2 * C}))


def rows_launches(L: int, M: int, kv_only: bool) -> int:
    """Kernels of one multi-position batch: the start, ten per layer (the
    last layer three when only its cache entries are needed), and the final
    residual add."""
    return 1 + 10 * (L - 1) + (3 if kv_only else 11)


def profile_rows(shape, model, local: int):
    """--profile-run --rows: the multi-position layer pass for ncu captures.
    A 256-position prompt in two batches, 16 exit steps (direct launches),
    then one re-pass of those 16 positions in one batch.  Prints the launch
    counts of each part."""
    from paper_2609_14144_gb300 import DEVICE, FORCE_EXIT_AT, OPT_GRAPHS, OPT_ROWS, Engine

    P, n = 2 * ROWS_MAX, REPASS_W
    eng = Engine(shape, model, max_ctx=P + n, device=local)
    eng.set_option(OPT_GRAPHS, 0)
    eng.set_option(OPT_ROWS, 1)
    eng.prefill(synth.prompt(shape, P))
    eng.decode_n(n, [0.5], schedule=np.full(n, FORCE_EXIT_AT(0), np.int8), where=DEVICE)
    eng.sync()
    n_rp = eng.repass(P, P + n)
    L, k = shape.n_layers, shape.readout_layers[0]
    prefill = rows_launches(L, ROWS_MAX, True) + rows_launches(L, P - ROWS_MAX, False) + 4
    decode = sum(step_launches(L, shape.readout_layers, 0, eng.persistent) for _ in range(n)) + 1
    repass = rows_launches(L - k, n, False)
    print(json.dumps({"prefill_launches": prefill, "decode_launches": decode, "repass_launches": repass,
                      "repassed": n_rp}))


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--no-sweep", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--profile-run", action="store_true", help="short decode for ncu captures")
    ap.add_argument("--eager", action="store_true", help="with --profile-run: direct launches, no graphs")
    ap.add_argument("--rows", action="store_true", help="with --profile-run: the multi-position layer pass")
    ap.add_argument("--workload", default=WORKLOAD, choices=sorted(synth.CONFIGS),
                    help="synthetic shape (the benchmark workload is 1.5b)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    globals()["WORKLOAD"] = args.workload
    rank, world, local = dist_setup()
    if args.profile_run:
        profile_run(args, local)
        return
    if args.impl == "reference":
        run_reference(args, rank, world)
    else:
        run_ours(args, rank, world, local)
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
