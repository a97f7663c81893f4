#!/usr/bin/env python3
"""Throughput of the DC-Leap denoise step on GB300.

A step is one pass of the whole hot path: re-mask the window, one bidirectional
forward over prompt + generation (embedding, 32 x {RMSNorm, QKV+RoPE GEMM, non-causal
attention, O GEMM + residual, RMSNorm, gate/up GEMM + SwiGLU, down GEMM + residual},
final RMSNorm, LM-head GEMM fused with softmax top-1/top-2), then the contiguous
commit / draft update / advance.  The default workload is the LLaDA-8B shape at batch 1,
prompt 256, generation 256, block 32, window 128, full recompute, with random-init bf16
weights (seed 1) and a random prompt.

Timed region: K steps (one CUDA-graph launch each) on the context stream, bracketed
by CUDA events, inputs resident in HBM; generations of the same prompt run back to
back (an on-device restart when a generation finishes), so `value` counts the tokens
committed in exactly those K steps.  Per-kernel times come from a second pass of the
same steps with timing events captured around every kernel.  `e2e` runs whole
generations through the public API (prompt from pinned host memory, result read back).

Under full recompute the line also carries `ms_per_step_at_p`: one step timed from the
trajectory's states at p - N = 0, M/4, M/2, 3M/4 (set back each time), so that the step
cost is read at fixed positions as well as over the trajectory.  With the key / value
cache it carries `ms_per_step_by_rows`: the trajectory's steps (each between CUDA events)
grouped by the rows they compute, median time and roofline fraction per row count.

--workload accept times the acceptance pass alone (dcl_accept on seeded bf16 logits
[64][32][126464], window 16) against the HBM roofline of the uncommitted logit rows it
must read.

--impl reference times the CPU oracle (tests' reference implementation) on a bounded
sample of the same step on the host cores.
"""
from __future__ import annotations

import argparse
import json
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

METRIC = "generated tokens/s and ms/denoise-step, LLaDA-8B shape, 1×GB300; % roofline"

WORKLOADS = {
    # LLaDA-8B shape, batch 1, prompt 256, gen 256, block 32, L = M/2, full recompute
    "llada8b": dict(shape="llada8b", batch=1, n_prompt=256, gen=256, block=32, window=128,
                    seed=1, lm_scale=12.0, tau_c=0.70, tau_d=0.98),
    # the same architecture, long generation: prompt 512, gen 1024, batch 1
    "llada8b-long": dict(shape="llada8b", batch=1, n_prompt=512, gen=1024, block=32, window=512,
                         seed=1, lm_scale=12.0, tau_c=0.70, tau_d=0.98),
    # the same, batch 8, full recompute
    "llada8b-long-b8": dict(shape="llada8b", batch=8, n_prompt=512, gen=1024, block=32, window=512,
                            seed=1, lm_scale=12.0, tau_c=0.70, tau_d=0.98),
    # Dream-7B shape (GQA 28 / 4 heads), batch 16, prompt 384, gen 512, full recompute
    "dream7b": dict(shape="dream7b", batch=16, n_prompt=384, gen=512, block=32, window=256,
                    seed=2, lm_scale=12.8, tau_c=0.70, tau_d=0.98),
    # the same three with the approximate prefix key / value cache (refresh every 32 positions)
    "llada8b-long-cache": dict(shape="llada8b", batch=1, n_prompt=512, gen=1024, block=32, window=512,
                               seed=1, lm_scale=12.0, tau_c=0.70, tau_d=0.98, cache=1),
    "llada8b-long-b8-cache": dict(shape="llada8b", batch=8, n_prompt=512, gen=1024, block=32, window=512,
                                  seed=1, lm_scale=12.0, tau_c=0.70, tau_d=0.98, cache=1),
    # the dual (prefix + suffix) cache: between refreshes only the current 32-position block
    "llada8b-long-dualcache": dict(shape="llada8b", batch=1, n_prompt=512, gen=1024, block=32, window=512,
                                   seed=1, lm_scale=12.0, tau_c=0.70, tau_d=0.98, cache=2),
    "llada8b-long-b8-dualcache": dict(shape="llada8b", batch=8, n_prompt=512, gen=1024, block=32, window=512,
                                      seed=1, lm_scale=12.0, tau_c=0.70, tau_d=0.98, cache=2),
    "dream7b-cache": dict(shape="dream7b", batch=16, n_prompt=384, gen=512, block=32, window=256,
                          seed=2, lm_scale=12.8, tau_c=0.70, tau_d=0.98, cache=1),
    "dream7b-dualcache": dict(shape="dream7b", batch=16, n_prompt=384, gen=512, block=32, window=256,
                              seed=2, lm_scale=12.8, tau_c=0.70, tau_d=0.98, cache=2),
    # the LLaDA-8B shape cut to 2 layers (~3 GB on the device): the same GEMM, attention and
    # LM-head launches as the full model, small enough for ncu captures with replay
    "llada8b-2l": dict(shape="llada8b-2l", batch=1, n_prompt=256, gen=256, block=32, window=128,
                       seed=1, lm_scale=12.0, tau_c=0.70, tau_d=0.98),
    # 2-layer test model (latency-bound)
    "tiny": dict(shape="tiny", batch=1, n_prompt=32, gen=64, block=32, window=32,
                 seed=0, lm_scale=40.0, tau_c=0.70, tau_d=0.98, oracle_whole=True),
    # the acceptance pass alone on given bf16 logits: 64 sequences x 32 block positions x
    # vocabulary 126464, window 16 (so that the draft region is exercised)
    "accept": dict(kind="accept", batch=64, positions=32, vocab=126464, window=16, seed=7,
                   tau_c=0.70, tau_d=0.98),
}


def _env_int(name, default):
    try:
        return int(os.environ.get(name, default))
    except ValueError:
        return default


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "bf16_tflops": float(p["bf16_tflops"]),
                "bf16_tflops_sustained": float(p.get("bf16_tflops_sustained", p["bf16_tflops"])),
                "source": "measured"}
    except (OSError, KeyError, ValueError):
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                "source": "fallback"}


def step_work(shape, B, N, M, rows=None, lm_rows=None, cached=False):
    """Algorithmic flops per step by kernel class, and the minimum HBM bytes of a step.

    Full recompute computes all B*T rows; with the key / value cache a step computes
    ``rows`` query rows (``lm_rows`` of them at generation positions), each attending to all
    T positions, and reads the stored keys / values of every layer."""
    T = N + M
    R = B * T if rows is None else rows
    R_lm = B * M if lm_rows is None else lm_rows
    d, H, G, hd, F, V = (shape.d_model, shape.n_heads, shape.n_kv_heads, shape.head_dim,
                         shape.ffn_dim, shape.vocab)
    L = shape.n_layers
    flops = {
        "gemm_qkv": 2.0 * R * d * (H + 2 * G) * hd,
        "gemm_o": 2.0 * R * H * hd * d,
        "gemm_gateup": 2.0 * R * d * 2 * F,
        "gemm_down": 2.0 * R * F * d,
        "attention": 4.0 * R * T * H * hd,
    }
    per_layer = dict(flops)
    total = {k: v * L for k, v in flops.items()}
    total["gemm_lmhead"] = 2.0 * R_lm * d * V
    w_layer = 2.0 * (d * (H + 2 * G) * hd + H * hd * d + 2 * F * d + F * d + 2 * d)
    bytes_ = L * w_layer + 2.0 * V * d + 2.0 * R * d + 2.0 * d
    if cached:
        bytes_ += L * 2.0 * 2.0 * B * T * G * hd  # stored keys and values read by the attention
    return per_layer, total, bytes_


def cached_rows(kper, N, M, block, dual=False):
    """Per step of a trajectory (per-row K values), the rows the cached step computes and
    its LM rows (the refresh rule of the key / value cache; with ``dual``, between
    refreshes only the current block)."""
    B = len(kper[0])
    T = N + M
    p = [N] * B
    pe_prev = [None] * B
    out = []
    for k in kper:
        rows = lm = 0
        for b in range(B):
            if p[b] >= T:
                continue
            pe = N + block * ((p[b] - N) // block)
            start = 0 if pe != pe_prev[b] else pe
            end = min(pe + block, T) if (dual and start) else T
            pe_prev[b] = pe
            rows += end - start
            lm += end - max(start, N)
            p[b] += int(k[b])
        out.append((rows, lm))
    return out


def steps_by_rows(rl, works, traj_ms, peaks):
    """Cached trajectories: the step time by the number of rows the step computes (all T
    positions at a refresh, the block-aligned suffix otherwise), median over the
    trajectory's steps with that row count, against the roofline of that step's own work
    (measured sustained bf16 peak, measured HBM copy rate)."""
    groups = {}
    for (rows, _), w, ms in zip(rl, works, traj_ms):
        g = groups.setdefault(rows, {"ms": [], "work": w})
        g["ms"].append(ms)
    out = []
    for rows in sorted(groups, reverse=True):
        g = groups[rows]
        flops = sum(g["work"][1].values())
        t_tensor = flops / (peaks["bf16_tflops_sustained"] * 1e12)
        t_hbm = g["work"][2] / (peaks["hbm_gbs"] * 1e9)
        ms = statistics.median(g["ms"])
        out.append({"rows": int(rows), "steps": len(g["ms"]), "ms": ms, "t_roof_ms": 1e3 * max(t_tensor, t_hbm),
                    "bound": "hbm" if t_hbm >= t_tensor else "tensor",
                    "frac": 1e3 * max(t_tensor, t_hbm) / ms if ms > 0 else None})
    return out


def k_histogram(kper):
    """{K: number of (step, row) pairs that committed K tokens} over a trajectory's per-row
    K values; rows that had finished (K = 0) are left out."""
    k = np.concatenate([np.asarray(v).ravel() for v in kper]) if kper else np.zeros(0, np.int64)
    k = k[k > 0]
    return {str(int(v)): int(n) for v, n in zip(*np.unique(k, return_counts=True))}


# ---------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid=None):
        self.uuid = uuid
        self.proc = None
        self.f = None

    def start(self):
        try:
            self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                   "-lms", "100"]
            if self.uuid:
                cmd += ["-i", self.uuid]
            self.proc = subprocess.Popen(cmd, stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.flush()
        self.f.seek(0)
        rows = [r.split(",") for r in self.f.read().strip().splitlines() if r.count(",") >= 8]
        self.f.close()
        os.unlink(self.f.name)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].strip().replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].strip().replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if "Active" in v and "Not" not in v})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


# ---------------------------------------------------------------------- oracle timing
def _layer_weights(shape, seed, layer):
    import synthetic as syn
    K = syn.TensorKind
    d, H, G, hd, F = shape.d_model, shape.n_heads, shape.n_kv_heads, shape.head_dim, shape.ffn_dim
    dims = {"attn_norm": (K.ATTN_NORM, (d,)), "wq": (K.WQ, (H * hd, d)), "wk": (K.WK, (G * hd, d)),
            "wv": (K.WV, (G * hd, d)), "wo": (K.WO, (d, H * hd)), "mlp_norm": (K.MLP_NORM, (d,)),
            "w_gate": (K.W_GATE, (F, d)), "w_up": (K.W_UP, (F, d)), "w_down": (K.W_DOWN, (d, F))}
    out = {}
    for name, (kind, shp) in dims.items():
        n = int(np.prod(shp))
        if kind in K.NORMS:
            v = syn.weight_values(seed, syn.tensor_id(kind, layer), 0, n, 0.0, 1.0)
        else:
            v = syn.weight_values(seed, syn.tensor_id(kind, layer), 0, n, 0.02)
        out[name] = v.reshape(shp)
    return out


def oracle_generation(wl, min_seconds=2.0):
    """The oracle's whole generation end to end (Algorithm 1, an fp64 forward at every
    step) on the workload's weights and prompts, repeated until `min_seconds` have passed:
    (seconds per generation, steps per generation, generations timed).  For the small
    shapes, whose generation takes well under a second."""
    import synthetic as syn
    from oracle import decode, model
    sh = syn.SHAPES[wl["shape"]]
    B, N, M = wl["batch"], wl["n_prompt"], wl["gen"]
    w = syn.model_weights(sh, wl["seed"], lm_head_scale=wl["lm_scale"])
    prompt = syn.prompt_ids(1000, B, N, sh.mask_id)
    cfg = decode.DecodeConfig(tau_commit=wl["tau_c"], tau_draft=wl["tau_d"], max_window=wl["window"],
                              block_len=wl["block"], gen_len=M)

    def predict(tokens):
        ids, p1, p2 = model.predict(sh, w, tokens)
        return ids[N:], p1[N:], p2[N:]
    n, t0 = 0, time.perf_counter()
    while True:
        out = decode.generate(predict, prompt, cfg, sh.mask_id, record=False)
        n += 1
        if time.perf_counter() - t0 >= min_seconds:
            break
    assert out["done"]
    return (time.perf_counter() - t0) / n, int(out["n_iter"]), n


def _step_margin(pr, x_in, p, K, N, L, tau_c, tau_d):
    """Smallest margin among the decisions of one oracle step of one row: |c - tau_c| over
    the window up to and including its first failure, |c - tau_d| over the draft region,
    and the top-1 / top-2 gap of every committed or drafted id."""
    ids, p1, p2 = pr[0], pr[1], pr[2]
    T = x_in.shape[0]
    c = np.zeros(T)
    gap = np.full(T, np.inf)
    c[N:], gap[N:] = p1, p1 - p2
    w = min(L, T - p)
    m = [np.abs(c[p:p + min(K + 1, w)] - tau_c).min(), gap[p:p + K].min()]
    if p + L < T:
        m.append(np.abs(c[p + L:] - tau_d).min())
        drafted = c[p + L:] > tau_d
        if drafted.any():
            m.append(gap[p + L:][drafted].min())
    return float(min(m))


def near_tie_study(ctx, dcl, shape, weights, N, M, L, tau_c, tau_d, seeds, tol=1e-3, drift=5e-2):
    """Whole generations of `seeds` random prompts on the GPU (step by step) and in the oracle
    (bf16 operands): per seed, whether the committed sequences are identical, else the
    oracle's smallest decision margin at the step where the two trajectories split:
    within `tol` (a near tie), within `drift` (inside the end-to-end confidence drift of the
    random model), or clear.  Returns the counts and the fraction of diverged seeds."""
    import synthetic as syn
    from oracle import decode, model
    T = N + M
    cfg = dcl.decode_config(tau_commit=tau_c, tau_draft=tau_d, max_window=L, gen_len=M)
    ocfg = decode.DecodeConfig(tau_commit=tau_c, tau_draft=tau_d, max_window=L, gen_len=M)
    predict = lambda t: model.predict(shape, weights, t, rows=slice(N, T), bf16_operands=True)  # noqa: E731
    out = {"seeds": len(seeds), "identical": 0, "split_near_tie": 0, "split_within_drift": 0, "split_clear": 0,
           "near_tie_margin": tol, "drift_margin": drift, "split_margins": []}
    for seed in seeds:
        prompt = syn.prompt_ids(3000 + seed, 1, N, shape.mask_id)
        ctx.set_prompt(prompt, cfg)
        states = []
        for _ in range(2 * M):
            x, p = ctx.get_state()
            states.append((x[0].copy(), int(p[0])))
            if p[0] >= T:
                break
            ctx.step()
        ref = decode.generate(predict, prompt, ocfg, shape.mask_id)
        p_o, split = N, None
        for s, xin in enumerate(ref["inputs"]):
            xg, pg = states[s] if s < len(states) else (None, -1)
            keep = (np.arange(T) < p_o) | (np.arange(T) >= p_o + L)  # not re-masked at this step
            if pg != p_o or not (xg == xin[0])[keep].all():
                split = s
                break
            p_o += int(ref["k"][s, 0])
        if split is None and (states[-1][0][N:] == ref["x"][0, N:]).all():
            out["identical"] += 1
            continue
        s = (split if split is not None else len(ref["inputs"])) - 1
        p_prev = p_o - int(ref["k"][s, 0]) if split is not None else p_o - int(ref["k"][s, 0])
        mg = _step_margin(ref["preds"][s][:, 0], ref["inputs"][s][0], p_prev, int(ref["k"][s, 0]), N, L, tau_c,
                          tau_d)
        out["split_margins"].append(mg)
        out["split_near_tie" if mg <= tol else "split_within_drift" if mg <= drift else "split_clear"] += 1
    out["fraction_diverged"] = 1.0 - out["identical"] / max(1, len(seeds))
    return out


class OracleSample:
    """A bounded sample of one step of the oracle: one transformer block over all T rows,
    and the LM head + confidence over 16 generation rows x 1/16 of the vocabulary; scaled
    to a step as n_layers x block + (B*M/16) x 16 x LM-head sample (an estimate of the
    step's time, not a timed step).  Both oracle legs credit a step one committed token per
    row, the least a step commits (the oracle cannot afford the 8B-shape trajectory that
    would give its real rate)."""

    RULE = ("ms_per_step is an estimate (the sample scaled to a step); tokens/s credits one committed token "
            "per row per step, the least a step commits")

    def __init__(self, wl):
        import synthetic as syn
        self.syn = syn
        self.shape = syn.SHAPES[wl["shape"]]
        self.wl = wl
        sh = self.shape
        B, N, M = wl["batch"], wl["n_prompt"], wl["gen"]
        self.T = N + M
        prompt = syn.prompt_ids(1000, 1, N, sh.mask_id)[0]
        tokens = np.concatenate([prompt, np.full(M, sh.mask_id, np.int32)])
        rows = {}
        for t in np.unique(tokens):
            rows[int(t)] = syn.weight_values(wl["seed"], syn.tensor_id(syn.TensorKind.EMBED, 0),
                                             int(t) * sh.d_model, sh.d_model, 0.02)
        self.h = np.stack([rows[int(t)] for t in tokens]).astype(np.float64)
        self.lw = _layer_weights(sh, wl["seed"], 0)
        self.vslice = max(1, sh.vocab // 16)
        std = float(np.float32(0.02) * np.float32(wl["lm_scale"]))
        self.lm = syn.weight_values(wl["seed"], syn.tensor_id(syn.TensorKind.LM_HEAD, 0), 0,
                                    self.vslice * sh.d_model, std).reshape(self.vslice, sh.d_model)
        self.lm_rows = min(16, B * M)
        self.scale_lm = (B * M / self.lm_rows) * (sh.vocab / self.vslice)
        self.B = B

    def step_seconds(self):
        from oracle import model
        sh = self.shape
        ang = model.rope_angles(self.T, sh.head_dim, sh.rope_theta)
        t0 = time.perf_counter()
        for _ in range(self.B):
            h1 = model.block(sh, self.lw, self.h, ang)
        t_block = time.perf_counter() - t0
        hn = model.rms_norm(h1[-self.lm_rows:], np.ones(sh.d_model), sh.rms_eps)
        t0 = time.perf_counter()
        model.confidence(model.logits({"lm_head": self.lm}, hn))
        t_lm = time.perf_counter() - t0
        return sh.n_layers * t_block + self.scale_lm * t_lm, t_block + t_lm

    def describe(self):
        sh = self.shape
        return (f"one transformer block over all {self.T} rows x batch {self.B} (x{sh.n_layers} layers) "
                f"+ LM head/confidence on {self.lm_rows} rows x {self.vslice} vocab rows "
                f"(x{self.scale_lm:.0f}); fp64 numpy, weight generation untimed")


def run_reference(args):
    rank = _env_int("RANK", 0)
    if rank != 0:
        return 0
    wl = WORKLOADS[args.workload]
    if wl.get("oracle_whole"):
        return run_reference_whole(args, wl)
    samp = OracleSample(wl)
    for _ in range(args.warmup):
        samp.step_seconds()
    secs, cpu = [], 0.0
    for _ in range(args.steps):
        s, c = samp.step_seconds()
        secs.append(s)
        cpu += c
    ms = 1e3 * statistics.mean(secs)
    tps = wl["batch"] * 1.0 / (ms / 1e3)  # one committed token per row per step (OracleSample.RULE)
    line = {
        "impl": "reference", "metric": METRIC, "value": tps, "unit": "tokens/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": _config(wl, args),
        "ms_per_step_is_estimate": True,
        "cpu_baseline": {"value": tps, "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
                         "sample": samp.describe() + "; " + OracleSample.RULE,
                         "cpu_seconds_timed": cpu},
        "e2e": {"value": tps, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


def run_reference_whole(args, wl):
    """The reference arm for the small shapes: every step is one whole oracle generation."""
    oracle_generation(wl, 0.0)  # warm-up
    secs, steps = [], 0
    for _ in range(args.steps):
        s, steps, _ = oracle_generation(wl, 0.0)
        secs.append(s)
    s = statistics.mean(secs)
    tokens = wl["batch"] * wl["gen"]
    tps = tokens / s
    line = {
        "impl": "reference", "metric": METRIC, "value": tps, "unit": "tokens/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * s / steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": _config(wl, args),
        "cpu_baseline": {"value": tps, "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
                         "sample": f"one whole generation per step ({steps} denoise steps, {tokens} tokens), "
                                   "fp64 numpy, weight generation untimed", "cpu_seconds_timed": sum(secs)},
        "e2e": {"value": tps, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


def _config(wl, args):
    return {"workload": f"{wl['shape']}-shape batch {wl['batch']}, prompt {wl['n_prompt']}, gen {wl['gen']}, "
                        f"block {wl['block']}, window {wl['window']}, tau_commit {wl['tau_c']}, "
                        f"tau_draft {wl['tau_d']}, "
                        + {0: "full recompute", 1: "approximate prefix key/value cache",
                           2: "dual (prefix + suffix) key/value cache"}[int(wl.get("cache", 0))],
            "global_batch": wl["batch"] * max(1, args.gpus), "seq_len": wl["n_prompt"] + wl["gen"],
            "parallelism": f"replicas{args.gpus}" if args.gpus > 1 else "single",
            "l2": _l2_note(wl)}


def _l2_note(wl):
    """How the timed steps treat the 129 MB L2: the large shapes stream every weight once per
    step; the small ones keep theirs in L2 (a latency figure, not a bandwidth one)."""
    import synthetic as syn
    _, _, bytes_ = step_work(syn.SHAPES[wl["shape"]], wl["batch"], wl["n_prompt"], wl["gen"])
    if bytes_ > 4 * 129e6:
        return "no flush needed: every step streams all weights (>> 129 MB L2)"
    return (f"not flushed: the {bytes_ / 1e6:.0f} MB of weights stay in the 129 MB L2; a latency-bound "
            "step, read as a latency figure")


def _allreduce(v, op, dist, device):
    """max or sum of a float over the ranks of `dist` (the value itself without one)."""
    if dist is None:
        return v
    import torch
    t = torch.tensor([v], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX if op == "max" else dist.ReduceOp.SUM)
    return float(t.item())


def aggregate_replicas(ms, tokens, e2e_s, dist=None, device="cuda"):
    """Whole-job numbers of N independent replicas (one per GPU, no data-path exchange):
    the slowest rank's timed window (ms), the tokens every rank committed in it, and the
    slowest rank's end-to-end generation time (s).  Timing only: the ranks share no data."""
    return (_allreduce(ms, "max", dist, device), _allreduce(tokens, "sum", dist, device),
            _allreduce(e2e_s, "max", dist, device))


def _gpu_uuid(torch, local):
    """The GPU's UUID as nvidia-smi names it (None when torch does not report one)."""
    try:
        uuid = str(torch.cuda.get_device_properties(local).uuid)
        return uuid if uuid.startswith("GPU-") else "GPU-" + uuid
    except Exception:
        return None


# ---------------------------------------------------------------------- our arm
def run_ours(args):
    import torch

    import synthetic as syn
    rank, world, local = _env_int("RANK", 0), _env_int("WORLD_SIZE", 1), _env_int("LOCAL_RANK", 0)
    dist = None
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    if local == 0:
        import __graft_entry__
        __graft_entry__.build()
    if dist:
        dist.barrier()
    import paper_2607_20467_gb300 as dcl

    wl = WORKLOADS[args.workload]
    shape = syn.SHAPES[wl["shape"]]
    B, N, M = wl["batch"], wl["n_prompt"], wl["gen"]
    T = N + M
    stream = torch.cuda.Stream()
    ctx = dcl.Context(shape, max_batch=B, max_seq=T, stream=stream.cuda_stream)
    ctx.init_random_weights(wl["seed"], 0.02, wl["lm_scale"], 0.0)
    prompt = syn.prompt_ids(1000 + rank, B, N, shape.mask_id)
    cached = int(wl.get("cache", 0))
    cfg = dcl.decode_config(tau_commit=wl["tau_c"], tau_draft=wl["tau_d"], max_window=wl["window"],
                            block_len=wl["block"], gen_len=M, kv_cache=cached)
    ctx.set_prompt(prompt, cfg)

    # one generation step by step: the trajectory (tokens committed per step) + warm-up.
    # Under full recompute the states at p - N = 0, M/4, M/2, 3M/4 (the slowest row; the
    # first state at or past each mark) are kept for the fixed-state step timings.
    marks = [] if cached else [0, M // 4, M // 2, 3 * M // 4]
    snaps = []
    ks, kper, traj_ms = [], [], []
    p_host = np.full(B, N, np.int64)
    while sum(ks) < B * M and len(ks) < 4 * M:
        if marks and int(p_host.min()) - N >= marks[0]:
            snaps.append(ctx.get_state())
            while marks and int(p_host.min()) - N >= marks[0]:
                marks.pop(0)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        ctx.step()
        e1.record(stream)
        _, p_new = ctx.get_state()  # (synchronises) K = the advance of p (contiguous commits)
        kr = (p_new.astype(np.int64) - p_host).astype(np.int32)
        traj_ms.append(e0.elapsed_time(e1))
        kper.append(kr.copy())
        ks.append(int(kr.sum()))
        p_host += kr
    S = len(ks)
    ctx.restart()
    for _ in range(args.warmup):
        ctx.step()
    torch.cuda.synchronize()

    def timed(nsteps, profiled=False):
        ctx.restart()
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        j = tokens = 0
        t0.record(stream)
        for _ in range(nsteps):
            if j == S:
                ctx.restart()
                j = 0
            ctx.step()
            tokens += ks[j]
            j += 1
        t1.record(stream)
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
        _, p = ctx.get_state()
        assert int((p - N).sum()) == sum(ks[:j]), "step trajectory did not replay deterministically"
        return t0.elapsed_time(t1), tokens

    sampler = ClockSampler(_gpu_uuid(torch, local))
    sampler.start()
    if args.profiler_range:
        torch.cuda.cudart().cudaProfilerStart()
    ms, tokens = timed(args.steps)
    if args.profiler_range:
        torch.cuda.cudart().cudaProfilerStop()
    clocks = sampler.stop()

    # per-kernel device times: the same steps with timing events around every kernel
    ctx.set_profiling(True)
    ms_prof, _ = timed(min(args.steps, max(3, S)))  # (n_prof steps)
    kern_ms, kern_kind = ctx.profile_last_step()
    ctx.set_profiling(False)

    # one step from each kept state (set_state, then one step between CUDA events), median
    # of 5: the step's cost at fixed positions, apart from the trajectory's dynamics
    at_p = []
    for xs, ps in snaps:
        t = []
        for _ in range(5):
            ctx.set_state(xs, ps)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            ctx.step()
            e1.record(stream)
            torch.cuda.synchronize()
            t.append(e0.elapsed_time(e1))
        at_p.append({"p_minus_n": int(ps.min()) - N, "ms": statistics.median(t)})

    # e2e through the public API: set_prompt (pinned host prompt) + generate (pinned out)
    pin_prompt = torch.from_numpy(prompt.copy()).pin_memory().numpy()
    pin_out = torch.zeros((B, M), dtype=torch.int32).pin_memory().numpy()
    e2e_s, e2e_steps = [], []
    for _ in range(args.e2e_iters):
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
        t = time.perf_counter()
        ctx.set_prompt(pin_prompt, cfg)
        _, st, _ = ctx.generate(max_steps=4 * M, out=pin_out)
        e2e_s.append(time.perf_counter() - t)
        e2e_steps.append(int(st.steps))
        assert st.done == 1

    # every step costs the same (full recompute), so a timed window of K steps is credited
    # the trajectory's average rate, B*M tokens per S steps: the window need not cover
    # whole generations for the value to equal whole-generation throughput
    per_step = B * M / S
    # (cached steps differ in cost: the window is credited the tokens it actually committed)
    ms_max, tokens_all, e2e_mean = aggregate_replicas(ms, tokens if cached else args.steps * per_step,
                                                      statistics.mean(e2e_s), dist, "cuda")
    peaks = _peaks()
    if cached:
        # the cached step's work varies (refresh or suffix): the mean over exactly the steps
        # timed (the window replays the trajectory from its start, wrapping at its end)
        rl = cached_rows(kper, N, M, wl["block"], dual=cached == 2)
        works = [step_work(shape, B, N, M, r, l, True) for r, l in rl]
        timed_works = [works[i % S] for i in range(args.steps)]
        per_layer = works[0][0]
        total_flops = {k: statistics.mean(w[1][k] for w in timed_works) for k in works[0][1]}
        step_bytes = statistics.mean(w[2] for w in timed_works)
        by_rows = steps_by_rows(rl, works, traj_ms, peaks)
    else:
        by_rows = None
        per_layer, total_flops, step_bytes = step_work(shape, B, N, M)

    # per-kernel table and the dominant kernel's roofline
    names = dcl.KERNEL_KINDS
    table = {}
    for t_ms, k in zip(kern_ms, kern_kind):
        e = table.setdefault(names[k], {"launches": 0, "ms": 0.0})
        e["launches"] += 1
        e["ms"] += float(t_ms)
    tot = sum(e["ms"] for e in table.values())
    for e in table.values():
        e["share"] = e["ms"] / tot if tot else 0.0
    # (the table is the last profiled step: with the cache, that step's own work)
    n_prof = min(args.steps, max(3, S))
    kern_flops = dict(works[(n_prof - 1) % S][1] if cached else total_flops)
    kern_flops["gemm_mlp"] = kern_flops["gemm_gateup"] + kern_flops["gemm_down"]  # (the fused MLP launch)
    gemms = {k: v for k, v in table.items() if k.startswith("gemm") and k in kern_flops}
    dom = max(gemms, key=lambda k: gemms[k]["ms"])
    avg_ms = gemms[dom]["ms"] / gemms[dom]["launches"]
    flops_launch = kern_flops[dom] / gemms[dom]["launches"]
    achieved = flops_launch / (avg_ms / 1e3) / 1e12
    peak = peaks["bf16_tflops_sustained"]
    for k, e in table.items():
        if k in kern_flops:
            e["tflops"] = kern_flops[k] / (e["ms"] / 1e3) / 1e12
    step_flops = sum(total_flops.values())
    ms_step = ms_max / args.steps
    t_roof = max(step_flops / (peak * 1e12), step_bytes / (peaks["hbm_gbs"] * 1e9))
    traffic = _traffic_from_profiles(dom)
    # the launch floor: a graph of as many empty dependent launches as a step has
    floor_ms = ctx.launch_floor(len(kern_ms), reps=200)

    # CPU oracle on a bounded sample (rank 0, one GPU only)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        if wl.get("oracle_whole"):
            s, steps_o, n = oracle_generation(wl)
            cpu = {"value": B * M / s, "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
                   "sample": f"whole generations end to end ({steps_o} denoise steps, {B * M} tokens each; "
                             f"{n} timed), fp64 numpy", "ms_per_step": 1e3 * s / steps_o,
                   "cpu_seconds_timed": s * n}
            # the same oracle generations against the GPU's on 32 prompts: how often and at
            # which decision margins the committed sequences part
            w_host = syn.model_weights(shape, wl["seed"], 0.02, wl["lm_scale"], 0.0)
            cpu["near_tie_divergence"] = near_tie_study(ctx, dcl, shape, w_host, N, M, wl["window"], wl["tau_c"],
                                                        wl["tau_d"], range(32))
        else:
            samp = OracleSample(wl)
            s, c = samp.step_seconds()
            cpu = {"value": B * 1.0 / s, "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
                   "sample": samp.describe() + "; " + OracleSample.RULE, "ms_per_step": 1e3 * s,
                   "ms_per_step_is_estimate": True, "cpu_seconds_timed": c,
                   "tokens_per_s_at_gpu_trajectory_rate": per_step / s}

    line = {
        "metric": METRIC, "value": tokens_all / (ms_max / 1e3), "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": f"synthetic: random-init bf16 weights (seed {wl['seed']}, LM head x{wl['lm_scale']}), "
                f"random prompts",
        "config": _config(wl, argparse.Namespace(gpus=world)),
        "steps_per_token": S / M,
        "trajectory_steps": S,
        "k_histogram": k_histogram(kper),
        "tokens_in_timed_window": tokens,
        "step_roofline": {"flops": step_flops, "bytes": step_bytes, "t_roof_ms": 1e3 * t_roof,
                          "frac": 1e3 * t_roof / ms_step, "peak_tflops": peak,
                          "peak_source": peaks["source"] + " sustained"},
        "roofline": {"kernel": dom, "bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak, "traffic": traffic,
                     "peak_source": f"{peaks['source']} bf16 sustained (kernel timed inside a long step)",
                     "avg_launch_ms": avg_ms, "flops_per_launch": flops_launch},
        "kernels": table,
        "ms_per_step_at_p": at_p or None,
        "ms_per_step_by_rows": by_rows,
        "ms_per_step_profiled": ms_prof / min(args.steps, max(3, S)),
        "gpu_launches": args.steps * len(kern_ms),
        "launch_floor": {"ms_per_graph": floor_ms, "launches_per_step": len(kern_ms),
                         "step_over_floor": ms_step / floor_ms,
                         "what": "a CUDA graph of as many empty kernels (dependent launches, as the step's) "
                                 "as one step launches"},
        "clocks": clocks,
        "e2e": {"value": world * B * M / e2e_mean, "unit": "tokens/s",
                "h2d_bytes_per_step": 4 * B * T + 12 * B + 4,
                "d2h_bytes_per_step": 4 * B * M + 8 * B + 4 * (statistics.mean(e2e_steps) + 1),
                "step": "one dcl_set_prompt + dcl_generate call (a whole generation)",
                "ms_per_generation": 1e3 * e2e_mean, "steps_per_generation": statistics.mean(e2e_steps)},
        "cpu_baseline": cpu,
    }
    if rank == 0:
        print(json.dumps(line))
    ctx.close()
    if dist:
        dist.destroy_process_group()
    return 0


# ---------------------------------------------------------------------- acceptance pass alone
ACCEPT_METRIC = ("uncommitted block positions decided/s by the acceptance pass on bf16 logits, 1×GB300; "
                 "% HBM roofline")


def _accept_config(wl, args):
    return {"workload": f"acceptance pass alone: bf16 logits [{wl['batch']}][{wl['positions']}][{wl['vocab']}] "
                        f"(top-1 probability from a Beta mixture, committed prefixes uniform in "
                        f"0..{wl['positions']}), window {wl['window']}, tau_commit {wl['tau_c']}, "
                        f"tau_draft {wl['tau_d']}",
            "global_batch": wl["batch"] * max(1, args.gpus), "seq_len": wl["positions"],
            "parallelism": f"replicas{args.gpus}" if args.gpus > 1 else "single",
            "l2": "no flush needed: every call streams the uncommitted logit rows (240 MB > 129 MB L2)"}


def _accept_data(wl, rank=0, nseq=None):
    """Seeded inputs of the acceptance pass (logits of the first `nseq` sequences only when
    given) and the number of uncommitted positions among those sequences."""
    import synthetic as syn
    V, P = wl["vocab"], wl["positions"]
    nseq = nseq or wl["batch"]
    only = None if nseq == wl["batch"] else {(b, i) for b in range(nseq) for i in range(P)}
    d = syn.accept_inputs(wl["seed"] + rank, wl["batch"], P, V, V - 1, rows=only)
    rows = int(np.clip(P - d["committed"][:nseq], 0, None).sum())
    return d, rows


def _accept_oracle_seconds(wl, d, nseq=None):
    """The oracle's acceptance pass over the first `nseq` sequences (all by default), one
    call (fp64 numpy); the bf16 -> float conversion is not timed."""
    import synthetic as syn
    from oracle import accept, decode
    nseq = nseq or wl["batch"]
    z = syn.bf16_to_f32(d["logits_bf16"][:nseq])
    cfg = decode.DecodeConfig(tau_commit=wl["tau_c"], tau_draft=wl["tau_d"], max_window=wl["window"],
                              gen_len=wl["positions"])
    t0 = time.perf_counter()
    accept.accept(z, d["committed"][:nseq], d["x"][:nseq], cfg, wl["window"])
    return time.perf_counter() - t0


def run_accept(args):
    """dcl_accept on the config's logits: K calls back to back on the context stream.

    A call is the two launches of the acceptance pass (softmax statistics of every
    uncommitted position, then the contiguous commit and drafts); its algorithmic bytes
    are the uncommitted logit rows, each read once.  Repeated calls see the same inputs
    and write the same outputs (K depends on the logits and the committed prefix only)."""
    import torch

    wl = WORKLOADS[args.workload]
    rank, world, local = _env_int("RANK", 0), _env_int("WORLD_SIZE", 1), _env_int("LOCAL_RANK", 0)
    dist = None
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    if local == 0:
        import __graft_entry__
        __graft_entry__.build()
    if dist:
        dist.barrier()
    import paper_2607_20467_gb300 as dcl

    B, P, V = wl["batch"], wl["positions"], wl["vocab"]
    d, rows = _accept_data(wl, rank)
    stream = torch.cuda.Stream()
    ctx = dcl.Context(None, 1, 1, stream=stream.cuda_stream)
    cfg = dcl.decode_config(tau_commit=wl["tau_c"], tau_draft=wl["tau_d"], max_window=wl["window"], gen_len=P)
    host_logits = torch.from_numpy(d["logits_bf16"].view(np.int16)).pin_memory()
    host_committed = torch.from_numpy(d["committed"]).pin_memory()
    host_x = torch.from_numpy(d["x"].copy()).pin_memory()
    with torch.cuda.stream(stream):
        logits = host_logits.to("cuda", non_blocking=True).view(torch.bfloat16)
        committed = host_committed.to("cuda", non_blocking=True)
        x = host_x.to("cuda", non_blocking=True)
        k = torch.full((B,), -1, dtype=torch.int32, device="cuda")
    stream.synchronize()

    for _ in range(args.warmup):
        ctx.accept(logits, committed, x, cfg, k)
    stream.synchronize()
    k_ref, x_ref = k.clone(), x.clone()
    torch.cuda.synchronize()

    if dist:
        dist.barrier()
    sampler = ClockSampler(_gpu_uuid(torch, local))
    sampler.start()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(args.steps):
        ctx.accept(logits, committed, x, cfg, k)
    t1.record(stream)
    torch.cuda.synchronize()
    clocks = sampler.stop()
    if dist:
        dist.barrier()
    ms = t0.elapsed_time(t1)
    assert torch.equal(k, k_ref) and torch.equal(x, x_ref), "repeated acceptance calls differ"

    # e2e: host logits / state in, K and x out, through the same call
    out_k = torch.zeros(B, dtype=torch.int32).pin_memory()
    out_x = torch.zeros((B, P), dtype=torch.int32).pin_memory()
    e2e = []
    for _ in range(args.e2e_iters):
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
        t = time.perf_counter()
        with torch.cuda.stream(stream):
            logits.view(torch.int16).copy_(host_logits, non_blocking=True)
            committed.copy_(host_committed, non_blocking=True)
            x.copy_(host_x, non_blocking=True)
            ctx.accept(logits, committed, x, cfg, k)
            out_k.copy_(k, non_blocking=True)
            out_x.copy_(x, non_blocking=True)
        stream.synchronize()
        e2e.append(time.perf_counter() - t)
    assert torch.equal(out_k, k_ref.cpu()) and torch.equal(out_x, x_ref.cpu())

    rows_all = _allreduce(float(rows * args.steps), "sum", dist, "cuda")
    ms_max = _allreduce(ms, "max", dist, "cuda")
    e2e_s = _allreduce(statistics.mean(e2e), "max", dist, "cuda")
    e2e_rows = _allreduce(float(rows), "sum", dist, "cuda")
    peaks = _peaks()
    ms_call = ms / args.steps
    algo_bytes = rows * V * 2
    achieved = algo_bytes / (ms_call / 1e3) / 1e9
    # DRAM bytes of the statistics launch as captured on this workload's seeded inputs (948
    # live rows); other inputs have other live rows, hence no captured figure
    traffic = _traffic_from_profiles("accept_stats", "kernels.cu") if rows == 948 else None

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        s = _accept_oracle_seconds(wl, d)
        cpu = {"value": rows / s, "unit": "positions/s", "cores": os.cpu_count(), "kind": "oracle",
               "sample": f"the whole workload once ({rows} uncommitted positions of {B * P}); fp64 numpy, "
                         "bf16 -> float conversion untimed", "ms_per_step": 1e3 * s}
    line = {
        "metric": ACCEPT_METRIC, "value": rows_all / (ms_max / 1e3), "unit": "positions/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_max / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": f"synthetic: seeded bf16 logits (seed {wl['seed']}), random drafts and committed prefixes",
        "config": _accept_config(wl, argparse.Namespace(gpus=world)),
        "uncommitted_positions": rows,
        "roofline": {"kernel": "accept (statistics + commit launches, timed together)", "bound": "hbm",
                     "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                     "frac": achieved / peaks["hbm_gbs"], "traffic": traffic,
                     "traffic_kernel": "accept_stats (the commit pass reads < 10 KB)",
                     "peak_source": f"{peaks['source']} HBM copy (kernel timed alone)",
                     "avg_launch_ms": ms_call, "bytes_per_launch": algo_bytes,
                     "t_roof_ms": 1e3 * algo_bytes / (peaks["hbm_gbs"] * 1e9)},
        "gpu_launches": 2 * args.steps,
        "clocks": clocks,
        "e2e": {"value": e2e_rows / e2e_s, "unit": "positions/s",
                "h2d_bytes_per_step": host_logits.numel() * 2 + 4 * B + 4 * B * P,
                "d2h_bytes_per_step": 4 * B + 4 * B * P,
                "step": "logits, committed prefixes and x copied in, one dcl_accept call, K and x copied out",
                "ms_per_step": 1e3 * e2e_s},
        "cpu_baseline": cpu,
    }
    if rank == 0:
        print(json.dumps(line))
    ctx.close()
    if dist:
        dist.destroy_process_group()
    return 0


def run_accept_reference(args):
    if _env_int("RANK", 0) != 0:
        return 0
    wl = WORKLOADS[args.workload]
    nseq = wl["batch"]  # the whole workload per step (~1 s of CPU work)
    d, rows = _accept_data(wl)
    for _ in range(args.warmup):
        _accept_oracle_seconds(wl, d, nseq)
    secs = [_accept_oracle_seconds(wl, d, nseq) for _ in range(args.steps)]
    s = statistics.mean(secs)
    v = rows / s
    line = {
        "impl": "reference", "metric": ACCEPT_METRIC, "value": v, "unit": "positions/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * s, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": _accept_config(wl, args),
        "cpu_baseline": {"value": v, "unit": "positions/s", "cores": os.cpu_count(), "kind": "oracle",
                         "sample": f"the whole workload per step ({nseq} sequences, {rows} uncommitted "
                                   "positions); fp64 numpy, bf16 -> float conversion untimed",
                         "cpu_seconds_timed": sum(secs)},
        "e2e": {"value": v, "unit": "positions/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


def _traffic_from_profiles(kernel, source="gemm_tc.cu"):
    """DRAM bytes per launch of `kernel` from the committed ncu summary (profiles/traffic.txt),
    or None when its source file (csrc/<source>) has changed since the counters were taken."""
    import hashlib
    try:
        with open(os.path.join(ROOT, "paper_2607_20467_gb300", "csrc", source), "rb") as f:
            sha = hashlib.sha256(f.read()).hexdigest()[:16]
        with open(os.path.join(ROOT, "profiles", "traffic.txt")) as f:
            for line in f:
                parts = line.split()
                if len(parts) >= 3 and parts[0] == kernel and not line.startswith("#"):
                    return int(parts[1]) if parts[2] == sha else None
    except (OSError, ValueError):
        pass
    return None


# Threshold / window grids of the paper's sensitivity ablations (App. F.1: tau_c at
# tau_d = 0.98, tau_d at tau_c = 0.70, the maximum window L), the tau_c grid with the
# entropy confidence (App. F.3 alternatives), and the samplers DC-Leap is contrasted with
# on the same kernels: the non-contiguous threshold rule (Eq. threshold_pd) in the
# semi-autoregressive block at the same thresholds, and the base sampler's low-confidence
# remasking (one token per step, the most confident masked position of the block).
SWEEPS = (
    [("tau_commit", dict(tau_c=t, tau_d=0.98, window=None, confidence=0)) for t in (0.65, 0.68, 0.70, 0.72, 0.75, 0.80)]
    + [("tau_draft", dict(tau_c=0.70, tau_d=t, window=None, confidence=0)) for t in (0.85, 0.88, 0.90, 0.92, 0.95, 0.98)]
    + [("window", dict(tau_c=0.70, tau_d=0.98, window=w, confidence=0)) for w in (32, 64, 96, 128)]
    + [("tau_commit_entropy", dict(tau_c=t, tau_d=0.98, window=None, confidence=1)) for t in (0.65, 0.70, 0.80)]
    + [("threshold_pd", dict(tau_c=t, tau_d=0.98, window=None, confidence=0, acceptance=1))
       for t in (0.65, 0.70, 0.80, 0.90, 0.95)]
    + [("low_confidence_remasking", dict(tau_c=1.0, tau_d=0.98, window=None, confidence=0, acceptance=1))]
)


def run_sweep(args):
    """Step counts and throughput over the ablation grids: whole generations through
    dcl_generate (host clock around it, on-device restart between runs), one JSON line
    per grid point.  Random weights: the curves show the decoding mechanics on this
    hardware, not the paper's accuracy / TPS (those need trained weights)."""
    import torch

    import synthetic as syn
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_20467_gb300 as dcl

    wl = WORKLOADS[args.workload]
    shape = syn.SHAPES[wl["shape"]]
    B, N, M = wl["batch"], wl["n_prompt"], wl["gen"]
    stream = torch.cuda.Stream()
    ctx = dcl.Context(shape, max_batch=B, max_seq=N + M, stream=stream.cuda_stream)
    ctx.init_random_weights(wl["seed"], 0.02, wl["lm_scale"], 0.0)
    prompt = syn.prompt_ids(1000, B, N, shape.mask_id)
    for name, pt in SWEEPS:
        window = pt["window"] or wl["window"]
        cfg = dcl.decode_config(tau_commit=pt["tau_c"], tau_draft=pt["tau_d"], max_window=window,
                                block_len=wl["block"], gen_len=M, kv_cache=int(wl.get("cache", 0)),
                                confidence=pt["confidence"], acceptance=pt.get("acceptance", 0))
        ctx.set_prompt(prompt, cfg)
        ctx.generate(max_steps=4 * M, out=False)  # warm-up (graph capture for this config)
        secs, st = [], None
        for _ in range(max(1, args.e2e_iters)):
            ctx.restart()
            torch.cuda.synchronize()
            t = time.perf_counter()
            _, st, _ = ctx.generate(max_steps=4 * M, out=False)
            secs.append(time.perf_counter() - t)
        sec = min(secs)
        print(json.dumps({"sweep": name, "workload": args.workload, "tau_commit": pt["tau_c"],
                          "tau_draft": pt["tau_d"], "window": window, "confidence": pt["confidence"],
                          "acceptance": "threshold_pd" if pt.get("acceptance") else "dcv",
                          "steps": int(st.steps), "tokens": int(st.tokens),
                          "steps_per_token": st.steps / max(1, st.tokens / B),
                          "ms_per_step": 1e3 * sec / max(1, st.steps), "tokens_per_s": st.tokens / sec,
                          "jpde_bound_per_token": st.jpde_bound / max(1, st.tokens)}), flush=True)
    ctx.close()
    return 0


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=sorted(WORKLOADS), default="llada8b")
    ap.add_argument("--e2e-iters", type=int, default=2)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--profiler-range", action="store_true",
                    help="bracket the timed steps with cudaProfilerStart / Stop (for a profiler started "
                         "with profiling off, e.g. ncu --profile-from-start off)")
    ap.add_argument("--sweep", action="store_true",
                    help="steps / throughput over the tau_c, tau_d, L (and entropy) grids, one JSON line each")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    accept_only = WORKLOADS[args.workload].get("kind") == "accept"
    if args.sweep:
        if accept_only:
            ap.error("--sweep runs the decoding workloads only")
        return run_sweep(args)
    if args.impl == "reference":
        return run_accept_reference(args) if accept_only else run_reference(args)
    return run_accept(args) if accept_only else run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
