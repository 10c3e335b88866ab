#!/usr/bin/env python3
"""Accepted tokens/s of KnapSpec self-speculative decoding on one GB300.

A step is one pass of the whole hot path on one sequence: gamma skip-masked
draft steps (a1), the gamma+1-row verify pass with greedy acceptance (a2, a3),
the history cosines (a4) and the knapsack mask selection (a5, re-solved every
step).  `value` = accepted tokens (a + 1 per step) / device time of K steps;
`e2e` = the same through ks_generate_speculative with host output buffers,
wall clock.  Weights and prompts are seeded synthetic inputs (random-init
model shapes, uniform random token ids).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload llama8b-4k]
  python bench.py --impl reference ...   # the CPU oracle, same metric
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2602_20217_gb300.configs import WORKLOADS  # noqa: E402

METRIC = "accepted tokens/sec at batch 1 on 1xGB300; decode-step HBM GB/s vs ~8 TB/s peak"
UNIT = "tokens/s"
DEFAULT_WORKLOAD = "qwen32b-64k"   # the largest configuration that fits one GPU


def chain_traffic(bytes_per_launch: float):
    """DRAM bytes (read + write) per chain launch, scaled from the committed ncu
    capture (traffic per algorithmic byte x this run's algorithmic bytes per
    launch), or None when the kernel's sources changed since the capture."""
    import hashlib
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            rec = json.load(f)["chain_kernel"]
        h = hashlib.sha256()
        for name in rec["source_files"]:
            with open(os.path.join(ROOT, name), "rb") as f:
                h.update(f.read())
        if h.hexdigest() != rec["source_sha256"]:
            return None
        return float(rec["traffic_per_algorithmic_byte"]) * bytes_per_launch
    except Exception:
        return None


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


# ------------------------------------------------------------ oracle arm
class OracleSample:
    """A bounded sample of one greedy decode token of the workload for the
    plain fp32 C++ oracle (one thread): one layer's Attn + MLP sublayers at
    the workload's context (a synthetic KV cache) and 1/32 of the LM-head
    rows; the token time scales them to all layers and the full vocabulary.
    The sample's weights and cache are seeded normal values of the workload's
    shapes (the oracle's operation count does not depend on the values)."""

    def __init__(self, workload: str, seed: int = 0):
        from dataclasses import replace
        from oracle import cxx
        from paper_2602_20217_gb300 import synth
        wl = WORKLOADS[workload]
        self.sh = sh = wl.shape
        rng = np.random.default_rng(seed)
        normal = lambda shape: (0.02 * rng.standard_normal(shape, dtype=np.float32))
        self.lm_rows = (sh.vocab + 31) // 32
        sample = replace(sh, n_layers=1, vocab=self.lm_rows, dtype="f32")
        shapes = synth.weight_shapes(sample)
        w = {k: (np.ones(v, np.float32) if k in synth.NORM_KINDS else normal(v)) for k, v in shapes["global"].items()}
        w["layers"] = [{k: (np.ones(v, np.float32) if k in synth.NORM_KINDS else normal(v))
                        for k, v in shapes["layer"].items()}]
        self.m = cxx.Model(sample, w)
        self.n = wl.prompt_len
        self.K = rng.standard_normal((sh.n_kv_heads, self.n + 1, sh.head_dim), dtype=np.float32)
        self.V = rng.standard_normal((sh.n_kv_heads, self.n + 1, sh.head_dim), dtype=np.float32)
        self.x = normal((1, sh.d_model)) * 50.0

    def token_seconds(self) -> float:
        t0 = time.perf_counter()
        x1 = self.m.attn_sublayer(0, self.x, [self.n], self.K, self.V)
        x2 = self.m.mlp_sublayer(0, x1)
        t1 = time.perf_counter()
        self.m.final_logits(x2)
        t2 = time.perf_counter()
        return self.sh.n_layers * (t1 - t0) + (self.sh.vocab / self.lm_rows) * (t2 - t1)


def run_oracle_arm(args, workload):
    """Runs in a child process; returns the mean token time over the timed samples."""
    smp = OracleSample(workload)
    samples = []
    for i in range(args.warmup + args.steps):
        t = smp.token_seconds()
        if i >= args.warmup:
            samples.append(t)
    return float(np.mean(samples))


_T0 = time.time()


def progress(msg: str):
    """One timestamped line on stderr per bench stage (the JSON line stays alone on stdout)."""
    print(f"[bench {time.time() - _T0:7.1f}s] {msg}", file=sys.stderr, flush=True)


def cpu_model() -> str:
    """The host CPU's model name (lscpu, else /proc/cpuinfo)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith(("model name", "cpu model")):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    return "unknown"


def cpu_baseline(workload: str, steps: int = 1, warmup: int = 0, timeout: float = 600.0) -> dict:
    """The plain fp32 C++ oracle, single-threaded, on a bounded sample (see
    oracle_sample_seconds), in a child process."""
    code = ("import sys, json; sys.path.insert(0, %r); import bench; "
            "print(json.dumps(bench.run_oracle_arm(type('A', (), {'steps': %d, 'warmup': %d})(), %r)))"
            % (ROOT, steps, warmup, workload))
    out = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, timeout=timeout)
    if out.returncode != 0:
        raise RuntimeError("oracle baseline failed: " + out.stderr[-2000:])
    t_token = float(out.stdout.strip().splitlines()[-1])
    wl = WORKLOADS[workload]
    sh = wl.shape
    return {"value": 1.0 / t_token, "unit": UNIT, "cores": 1, "cpu_model": cpu_model(), "kind": "oracle",
            "sample": (f"plain fp32 C++ oracle (oracle/cpp, one thread), greedy decode token at "
                       f"{wl.prompt_len} context: one layer's Attn+MLP (synthetic KV cache) x {sh.n_layers} layers "
                       f"+ 1/32 of the LM-head rows x 32; {steps} timed sample(s) after {warmup} untimed; every "
                       f"emitted token counts as accepted")}


def reference_arm(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    wl = args.workload
    cb = cpu_baseline(wl, steps=args.steps, warmup=args.warmup)
    line = {"metric": METRIC, "value": cb["value"], "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 / cb["value"], "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "impl": "reference",
            "config": {"workload": wl, "prompt": WORKLOADS[wl].prompt_len},
            "cpu_baseline": cb,
            "e2e": {"value": cb["value"], "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------- GPU arm
class ClockSampler:
    def __init__(self, path):
        self.path = path
        self.proc = None

    def __enter__(self):
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={q}", "--format=csv,noheader,nounits",
                                          "-lms", "200"], stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(5)
            except Exception:
                self.proc.kill()
            self.f.close()

    def summary(self, gpu_index: int):
        try:
            rows = [l.split(",") for l in open(self.path).read().strip().splitlines()]
        except Exception:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        rows = [[c.strip() for c in r] for r in rows if r and r[0].strip() == str(gpu_index)]
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if len(r) > 5 + i and r[5 + i] == "Active"})
        return {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


def attention_ms(shape, n: int, seed: int = 0) -> float:
    """Per-launch time (ms, CUDA events) of the split-KV attention kernel of a
    greedy step at context n, on a one-layer model with the workload's
    attention shape (the kernel's time depends on the heads, head size and
    context, not on the model's depth)."""
    from dataclasses import replace
    import torch
    from paper_2602_20217_gb300 import knapspec as ks, synth
    from paper_2602_20217_gb300.configs import truncated
    from paper_2602_20217_gb300.model import Model
    sh = replace(truncated(shape, 1), vocab=1024)
    m = Model(sh, max_seq=n + 32, seed=seed)
    m.prefill(synth.prompt_tokens(sh, n, seed=1))
    k = ks.KLASS["attn"]
    ks.ks_kernel_timing(m.h, k, True)
    m.decode_greedy(3)
    ks.ks_kernel_timing(m.h, k, False)
    ks.ks_kernel_timing(m.h, k, True)
    m.decode_greedy(9)
    cnt, ms = ks.ks_kernel_time(m.h, k)
    ks.ks_kernel_timing(m.h, k, False)
    m.close()
    del m
    torch.cuda.empty_cache()
    return ms / max(1, cnt)


def reduce_over_ranks(ms: float, tokens: float, dist=None, device="cpu"):
    """Replicas: the job's time is the slowest rank's, its tokens the sum
    over ranks.  Returns (max ms, total tokens)."""
    import torch
    a = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    b = torch.tensor([float(tokens)], dtype=torch.float64, device=device)
    if dist is not None:
        dist.all_reduce(a, op=dist.ReduceOp.MAX)
        dist.all_reduce(b, op=dist.ReduceOp.SUM)
    return float(a[0]), float(b[0])


def gpu_arm(args):
    import torch
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    from paper_2602_20217_gb300 import build, knapspec as ks, synth
    from paper_2602_20217_gb300.model import Model
    build.build()

    wl = WORKLOADS[args.workload]
    sh = wl.shape
    gamma = args.gamma or wl.gammas[len(wl.gammas) // 2]
    prompt = synth.prompt_tokens(sh, wl.prompt_len, seed=wl.prompt_seed)
    g_max = max(gamma, int(args.tpt_max_gamma)) if args.policy == "tpt" or args.sweep else gamma
    max_seq = wl.prompt_len + (max(args.steps, args.warmup) + 2) * (g_max + 1) + (args.e2e_tokens or wl.new_tokens) + 64
    t0 = time.time()
    model = Model(sh, max_seq=max_seq, seed=wl.weight_seed)
    torch.cuda.synchronize()
    t_setup = time.time() - t0
    stream, h = model.stream, model.h

    def prefill():
        t = time.time()
        model.prefill(prompt)
        torch.cuda.synchronize()
        return time.time() - t

    def rewind():   # back to the post-prefill state; the prompt's KV cache is reused
        model.rewind()
        torch.cuda.synchronize()

    # Latency model of App. C measured on this GPU at the prompt's context:
    # c1 = MLP sublayer (gate/up + down), c3 = the Attn sublayer's
    # context-independent kernels (QKV, query prep, merge, O-proj), c2 =
    # attention-kernel time / context length.
    progress("model created; prefill")
    t_prefill = prefill()
    progress("prefill done; latency model")
    split = [k for name, k in ks.KLASS.items() if name != "chain"]   # one projection per launch
    for k in split:                  # untimed first launches of every kernel in that mode
        ks.ks_kernel_timing(h, k, True)
    model.decode_greedy(3)
    rewind()
    for k in split:                  # disabling resets the class's counters; re-enable to time
        ks.ks_kernel_timing(h, k, False)
        ks.ks_kernel_timing(h, k, True)
    model.decode_greedy(8)
    kt = {name: ks.ks_kernel_time(h, k) for name, k in ks.KLASS.items() if name != "chain"}
    for k in split:
        ks.ks_kernel_timing(h, k, False)
    per = lambda name: kt[name][1] / max(1, kt[name][0])
    c1 = per("gateup") + per("down")
    fixed = per("qkv") + per("prep") + per("merge") + per("oproj")
    # App. C's profiling sweep: the attention kernel's time at four context
    # lengths (a one-layer model with this attention shape, R = 1), fitted
    # with the fixed Attn-sublayer kernels by least squares (ks_fit_latency)
    progress("latency sweep")
    sweep_n = [max(256, wl.prompt_len // 8), max(512, wl.prompt_len // 4), max(1024, wl.prompt_len // 2),
               wl.prompt_len]
    sweep_t = [attention_ms(sh, n) for n in sweep_n]
    lat = ks.ks_fit_latency(sweep_n, [fixed + t for t in sweep_t], [c1])
    _keep = None
    c2, c3 = lat.c2, lat.c3

    tpt_d = int(args.tpt_max_gamma)   # D of Alg. 2: the longest draft the grid search may pick

    def params(max_steps):
        if args.policy == "tpt":
            return ks.KsSpecParams(gamma, 2, None, lat, 0.0, int(args.tpt_every), int(max_steps),
                                   int(args.tpt_candidates), tpt_d, float(args.tau_conf))
        return ks.KsSpecParams(gamma, 1, None, lat, float(args.budget_frac), int(args.resolve_every),
                               int(max_steps), 0, 0, float(args.tau_conf))

    # warm-up
    progress("warm-up")
    rewind()
    ks.ks_generate_speculative(h, params(args.warmup), 1 << 30)
    # timed region: exactly K speculation steps, device time on the model's
    # stream, no instrumentation (kernels overlap through programmatic
    # dependent launch as in normal use)
    rewind()
    launches0 = ks.ks_launch_count(h)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    clk_dir = args.clocks_dir or tempfile.gettempdir()   # the raw nvidia-smi samples
    clk_path = os.path.join(clk_dir, f"ks_clocks_rank{rank}.csv")
    clocks = ClockSampler(clk_path)
    with clocks:
        torch.cuda.nvtx.range_push("timed")  # lets a profiler capture exactly these steps
        ev0.record(stream)
        _, st, acc = ks.ks_generate_speculative(h, params(args.steps), 1 << 30)
        ev1.record(stream)
        torch.cuda.synchronize()
        torch.cuda.nvtx.range_pop()
    if dist:
        dist.barrier()
    ms = ev0.elapsed_time(ev1)
    launches = ks.ks_launch_count(h) - launches0
    tokens = int(st.steps + st.accepted)

    # the same K steps again with CUDA events around every chain-kernel
    # launch: its per-launch duration for the roofline object (the events
    # serialise the launches, so this pass is slower than the timed one)
    progress("instrumented pass of the same steps")
    rewind()
    ks.ks_kernel_timing(h, ks.KLASS["chain"], True)
    i0 = torch.cuda.Event(enable_timing=True)
    i1 = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    i0.record(stream)
    _, st_i, _ = ks.ks_generate_speculative(h, params(args.steps), 1 << 30)
    i1.record(stream)
    torch.cuda.synchronize()
    ms_instr = i0.elapsed_time(i1)
    ch_n, ch_ms = ks.ks_kernel_time(h, ks.KLASS["chain"])
    ch_bytes = ks.ks_kernel_bytes(h, ks.KLASS["chain"])
    ks.ks_kernel_timing(h, ks.KLASS["chain"], False)
    assert int(st_i.steps + st_i.accepted) == tokens, "the instrumented pass decoded differently"

    e2e_tokens = args.e2e_tokens or wl.new_tokens
    # e2e: the public call with host output buffers, wall clock, for a
    # generation job of e2e_tokens tokens (the prompt already prefilled)
    rewind()
    h2d0, d2h0 = ks.ks_transfer_bytes(h)
    t0 = time.perf_counter()
    progress("end-to-end job")
    out, est, eacc = ks.ks_generate_speculative(h, params(0), e2e_tokens)
    e2e_s = time.perf_counter() - t0
    h2d1, d2h1 = ks.ks_transfer_bytes(h)
    e2e_tok = int(est.steps + est.accepted)
    # the same library's plain greedy decode of the same job, wall clock
    rewind()
    t0 = time.perf_counter()
    progress("greedy job")
    ar = ks.ks_decode_greedy(h, e2e_tokens)
    ar_s = time.perf_counter() - t0
    lossless = bool(np.array_equal(out, ar))
    # and on the device clock, next to `value`
    rewind()
    g0 = torch.cuda.Event(enable_timing=True)
    g1 = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    g0.record(stream)
    ks.ks_decode_greedy(h, e2e_tokens)
    g1.record(stream)
    torch.cuda.synchronize()
    ar_dev = (e2e_tokens - 1) / (g0.elapsed_time(g1) * 1e-3)
    progress("greedy job done")

    sweep = []
    if args.sweep:
        # accepted tokens/s (device time) of e2e_tokens-token jobs over a grid
        # of knapsack budgets and draft lengths, next to the greedy decode
        def timed(fn):
            rewind()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            r = fn()
            e1.record(stream)
            torch.cuda.synchronize()
            return r, e0.elapsed_time(e1) * 1e-3
        _, t_ar = timed(lambda: ks.ks_decode_greedy(h, e2e_tokens))
        sweep.append({"policy": "greedy", "tokens_per_s": (e2e_tokens - 1) / t_ar})
        for g in sorted({int(x) for x in args.sweep_gammas.split(",")}):
            for bf in [float(x) for x in args.sweep_budgets.split(",")]:
                p = ks.KsSpecParams(g, 1, None, lat, bf, int(args.resolve_every), 0)
                (o, sst, _a), t = timed(lambda: ks.ks_generate_speculative(h, p, e2e_tokens))
                n_tok = int(sst.steps + sst.accepted)
                sweep.append({"gamma": g, "budget_frac": bf, "tokens_per_s": n_tok / t,
                              "vs_greedy": (n_tok / t) / ((e2e_tokens - 1) / t_ar),
                              "alpha": float(sst.accepted) / max(1, sst.drafted),
                              "tokens_per_step": n_tok / max(1, sst.steps),
                              "skipped_attn_mlp": [int(sst.attn_skipped), int(sst.mlp_skipped)]})
        # the TPT stage (Alg. 2) picks the layer set and gamma itself
        p = ks.KsSpecParams(gamma, 2, None, lat, 0.0, int(args.tpt_every), 0, int(args.tpt_candidates), tpt_d)
        (o, sst, _a), t = timed(lambda: ks.ks_generate_speculative(h, p, e2e_tokens))
        n_tok = int(sst.steps + sst.accepted)
        sweep.append({"policy": f"tpt every {args.tpt_every} steps, K {args.tpt_candidates}, D {tpt_d}",
                      "tokens_per_s": n_tok / t, "vs_greedy": (n_tok / t) / ((e2e_tokens - 1) / t_ar),
                      "alpha": float(sst.accepted) / max(1, sst.drafted),
                      "mean_gamma": float(sst.drafted) / max(1, sst.steps),
                      "tokens_per_step": n_tok / max(1, sst.steps),
                      "skipped_attn_mlp": [int(sst.attn_skipped), int(sst.mlp_skipped)]})
        # the dynamic drafting exit of Sec. 3.5 (tau_conf 0.7) on the default knapsack policy
        p = ks.KsSpecParams(gamma, 1, None, lat, float(args.budget_frac), int(args.resolve_every), 0, 0, 0, 0.7)
        (o, sst, _a), t = timed(lambda: ks.ks_generate_speculative(h, p, e2e_tokens))
        n_tok = int(sst.steps + sst.accepted)
        sweep.append({"policy": f"knapsack, gamma {gamma} max, budget {args.budget_frac}, dynamic exit tau_conf 0.7",
                      "tokens_per_s": n_tok / t, "vs_greedy": (n_tok / t) / ((e2e_tokens - 1) / t_ar),
                      "alpha": float(sst.accepted) / max(1, sst.drafted),
                      "drafts_per_step": float(sst.drafted) / max(1, sst.steps),
                      "tokens_per_step": n_tok / max(1, sst.steps)})
        # Alg. 1 (hidden-state DP, tau 0.5) + the Eq. 3 grid on a filled history, then the
        # e2e job decoded with the (S*, gamma*) it picks
        rewind()
        ks.ks_generate_speculative(h, ks.KsSpecParams(gamma, 1, None, lat, float(args.budget_frac),
                                                      int(args.resolve_every), 6), 1 << 20)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        dmask, dgamma, dtpt, djs, dalphas, dcands = model.select_dp((lat, _keep), tpt_d, tau=0.5, max_states=128,
                                                                    max_rows=32)
        dp_s = time.perf_counter() - t0
        dm = np.ascontiguousarray(dmask, np.uint8)
        p = ks.KsSpecParams(int(dgamma), 0, dm.ctypes.data_as(ks.C.POINTER(ks.C.c_uint8)), lat, 0.0, 1, 0)
        (o, sst, _a), t = timed(lambda: ks.ks_generate_speculative(h, p, e2e_tokens))
        n_tok = int(sst.steps + sst.accepted)
        sweep.append({"policy": f"hidden-state DP (Alg. 1, tau 0.5) + TPT grid (D {tpt_d}), selected once",
                      "dp_seconds": dp_s, "dp_candidates": int(len(djs)), "gamma": int(dgamma),
                      "skipped_attn_mlp": [int(np.sum(dmask[0::2] == 0)), int(np.sum(dmask[1::2] == 0))],
                      "tokens_per_s": n_tok / t, "vs_greedy": (n_tok / t) / ((e2e_tokens - 1) / t_ar),
                      "alpha": float(sst.accepted) / max(1, sst.drafted),
                      "tokens_per_step": n_tok / max(1, sst.steps)})
        # Eq. 3's prediction for the DP's best candidates (each at its best
        # gamma, the fitted latency model at the prompt's context, times in
        # ms) next to the tokens/s their jobs reach
        ta, tm = c2 * wl.prompt_len + c3, c1

        def predicted(mask_c, alpha, g):
            e = sum(alpha ** i for i in range(g + 1))
            td = int(np.sum(mask_c[0::2])) * ta + int(np.sum(mask_c[1::2])) * tm
            return 1e3 * e / (g * td + sh.n_layers * (ta + tm))
        ranked = sorted(((max(predicted(dcands[i], float(dalphas[i]), g) for g in range(1, tpt_d + 1)),
                          max(range(1, tpt_d + 1), key=lambda g: predicted(dcands[i], float(dalphas[i]), g)), i)
                         for i in range(len(djs))), reverse=True)
        checks = []
        for pred, g, i in ranked[:3]:
            mc = np.ascontiguousarray(dcands[i], np.uint8)
            p = ks.KsSpecParams(int(g), 0, mc.ctypes.data_as(ks.C.POINTER(ks.C.c_uint8)), lat, 0.0, 1, 0)
            (o, sst, _a), t = timed(lambda: ks.ks_generate_speculative(h, p, e2e_tokens))
            n_tok = int(sst.steps + sst.accepted)
            checks.append({"skipped_weight": int(djs[i]), "gamma": int(g), "alpha_hat": float(dalphas[i]),
                           "alpha": float(sst.accepted) / max(1, sst.drafted),
                           "predicted_tokens_per_s": pred, "tokens_per_s": n_tok / t})
        sweep.append({"policy": "Eq. 3 prediction vs measurement for the DP's three best candidates",
                      "candidates": checks, "greedy_predicted_tokens_per_s": 1e3 / (sh.n_layers * (ta + tm))})
        # sampling mode (Sec. 2.1; nucleus sampling with T 0.7, top-k 50, top-p 0.95 as in Sec. 4)
        p = ks.KsSpecParams(gamma, 1, None, lat, float(args.budget_frac), int(args.resolve_every), 0, 0, 0, 0.0,
                            ks.sampling(0.7, 50, 0.95, 12345))
        (o, sst, _a), t = timed(lambda: ks.ks_generate_speculative(h, p, e2e_tokens))
        n_tok = int(sst.steps + sst.accepted)
        sweep.append({"policy": f"knapsack, gamma {gamma}, budget {args.budget_frac}, sampling T 0.7 top-k 50 top-p 0.95",
                      "tokens_per_s": n_tok / t, "vs_greedy": (n_tok / t) / ((e2e_tokens - 1) / t_ar),
                      "alpha": float(sst.accepted) / max(1, sst.drafted),
                      "tokens_per_step": n_tok / max(1, sst.steps)})

    ms_max, tok_all = reduce_over_ranks(ms, tokens, dist, "cuda")

    if rank == 0:
        peak, peak_kind = peaks()
        # dominant kernel: the chained projections; algorithmic bytes = the
        # weight bytes of the projections each launch ran
        achieved = ch_bytes / (ch_ms * 1e-3) / 1e9 if ch_ms > 0 else 0.0
        # second kernel: split-KV attention of the greedy passes that calibrated
        # the latency model (R = 1, contexts prompt_len .. prompt_len + 7, CUDA
        # events around each launch); algorithmic bytes = the layer's K and V
        # up to the row's position
        n_ctx = wl.prompt_len + 4.5
        kv_bytes = 2.0 * sh.n_kv_heads * n_ctx * sh.head_dim * (2 if sh.dtype == "bf16" else 4)
        t_attn = per("attn") * 1e-3
        attn_roof = {"bound": "hbm", "achieved": kv_bytes / t_attn / 1e9 if t_attn > 0 else 0.0, "peak": peak,
                     "unit": "GB/s", "frac": (kv_bytes / t_attn / 1e9) / peak if t_attn > 0 else 0.0,
                     "kernel": "attn_bf16_kernel (R = 1, one launch per layer)", "bytes_per_launch": kv_bytes,
                     "us_per_launch": per("attn") * 1e3, "context": n_ctx}
        line = {
            "metric": METRIC, "value": tok_all / (ms_max * 1e-3), "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_max / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": sh.dtype,
            "data": "synthetic (seeded random-init weights, uniform random prompt ids)",
            "config": {"workload": wl.name, "prompt": wl.prompt_len, "gamma": gamma,
                       "policy": ((f"knapsack re-solved every {args.resolve_every} step(s), "
                                  f"budget {args.budget_frac} of sum w") if args.policy == "knapsack" else
                                 (f"TPT stage every {args.tpt_every} step(s), K {args.tpt_candidates}, "
                                  f"D {tpt_d}"))
                                 + (f", dynamic exit tau_conf {args.tau_conf}" if args.tau_conf > 0 else ""),
                       "l2": (f"inputs larger than L2 (each step streams "
                              f"{(sh.n_layers * (sh.attn_weight_bytes() + sh.mlp_weight_bytes()) + sh.lm_head_bytes()) / 1e9:.1f} GB of weights)"),
                       "parallelism": f"replicas x{world}"},
            "tokens": tokens, "mean_tokens_per_step": tokens / max(1, st.steps),
            "alpha": float(st.accepted) / max(1, st.drafted),
            "mean_gamma": float(st.drafted) / max(1, st.steps),
            "mask_skipped": {"attn": int(st.attn_skipped), "mlp": int(st.mlp_skipped)},
            "ar_tokens_per_s": (e2e_tokens - 1) / ar_s,
            "spec_vs_ar_e2e": (e2e_tok / e2e_s) / ((e2e_tokens - 1) / ar_s),
            "ar_tokens_per_s_device": ar_dev,
            "spec_vs_ar_device": (tok_all / (ms_max * 1e-3)) / ar_dev,
            "lossless_vs_ar": lossless,
            "latency_model_ms": {"c1": c1, "c2": c2, "c3": c3,
                                 "fit": "App. C least squares over attention at n = " + ",".join(map(str, sweep_n)),
                                 "attention_ms_at_n": [round(t, 5) for t in sweep_t], "fixed_attn_kernels_ms": fixed},
            "prefill_s": t_prefill, "setup_s": t_setup,
            "e2e": {"value": e2e_tok / e2e_s, "unit": UNIT,
                    "h2d_bytes_per_step": (h2d1 - h2d0) / max(1, est.steps),
                    "d2h_bytes_per_step": (d2h1 - d2h0) / max(1, est.steps)},
            "gpu_launches": launches,
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak,
                         "traffic": chain_traffic(ch_bytes / max(1, ch_n)),
                         "kernel": "chain_kernel (chained projections)", "peak_source": peak_kind,
                         "launches_timed": ch_n, "bytes_per_launch": ch_bytes / max(1, ch_n),
                         "timing": "CUDA events around each launch, in a second pass of the same steps",
                         "time_share": ch_ms / ms_instr, "instrumented_ms_per_step": ms_instr / args.steps},
            "kernels_us": {k: round(1e3 * v[1] / max(1, v[0]), 2) for k, v in kt.items()},
            "attention_roofline": attn_roof,
            "clocks": clocks.summary(local),
        }
        if sweep:
            line["sweep_device_time"] = sweep
        if not args.no_cpu_baseline and world == 1:
            try:
                progress("oracle baseline")
                line["cpu_baseline"] = cpu_baseline(wl.name)
            except Exception as e:  # reported, never hidden
                line["cpu_baseline"] = {"error": str(e)[:300]}
        print(json.dumps(line), flush=True)
    model.close()
    if dist:
        dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=48)
    ap.add_argument("--warmup", type=int, default=4)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(WORKLOADS))
    ap.add_argument("--gamma", type=int, default=0)
    ap.add_argument("--budget-frac", dest="budget_frac", type=float, default=0.8)
    ap.add_argument("--resolve-every", dest="resolve_every", type=int, default=1)
    ap.add_argument("--e2e-tokens", dest="e2e_tokens", type=int, default=0,
                    help="tokens of the end-to-end and greedy jobs (default: the workload's generation length)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--policy", default="knapsack", choices=["knapsack", "tpt"],
                    help="mask policy of the timed steps: knapsack at --budget-frac, or the TPT stage")
    ap.add_argument("--tpt-every", dest="tpt_every", type=int, default=8)
    ap.add_argument("--tpt-candidates", dest="tpt_candidates", type=int, default=8)
    ap.add_argument("--tau-conf", dest="tau_conf", type=float, default=0.0,
                    help="dynamic drafting exit threshold (Sec. 3.5); 0 drafts gamma tokens every step")
    ap.add_argument("--tpt-max-gamma", dest="tpt_max_gamma", type=int, default=10,
                    help="D of Alg. 2 (1..15; the paper's is 10)")
    ap.add_argument("--clocks-dir", dest="clocks_dir", default="",
                    help="directory for the raw clock samples of the timed region (default: the temp dir)")
    ap.add_argument("--sweep", action="store_true",
                    help="also time jobs over a grid of knapsack budgets and draft lengths")
    ap.add_argument("--sweep-budgets", dest="sweep_budgets", default="0.4,0.5,0.6,0.7,0.8")
    ap.add_argument("--sweep-gammas", dest="sweep_gammas", default="2,4,6")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        reference_arm(args)
    else:
        gpu_arm(args)


if __name__ == "__main__":
    main()
