"""Benchmark of the SD^2 hot path: one draft-and-verify iteration (steering, k drafter steps, the
verifier over k+1 rows, acceptance and rollback) per step, on synthetic inputs.

Default workload: a Llama-3-8B-shaped verifier with a Llama-3.2-1B-shaped drafter, batch 1,
prompt 512 uniform-random ids, k = 5, T = 1.0 (random-init bf16 weights N(0, 0.02^2)).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--workload NAME]
  python bench.py --sweep      # the kernel sweep: acceptance grid, steering, 16K-context verify

Prints one JSON line. `value` is emitted tokens per second per sequence (N > 1: summed over the
N independent replicas). The reference arm times the CPU oracle on a bounded slice of the same
workload (a few decoder layers, scaled to the full depth).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import torch  # noqa: E402

from paper_2511_09844_gb300 import workloads as W  # noqa: E402

METRIC = "steered-SD emitted tokens/sec/sequence at 1 GB300; verify-step HBM GB/s vs 8 TB/s"
NOMINAL_HBM_GBS = 8000.0


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=32)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="llama8b_1b", choices=sorted(W.WORKLOADS))
    ap.add_argument("--seed", type=int, default=1234)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extras", action="store_true",
                    help="leave out the other configurations' blocks (batch 16, Qwen pair, sweep corners, 16K verify)")
    ap.add_argument("--depth", default=None,
                    help="profiling aid: 'LV,LD' keeps the first LV verifier and LD drafter layers of the "
                         "workload (same widths, context and batch) so that an ncu capture holds a few GB; the "
                         "JSON line's config names the depth")
    ap.add_argument("--steer-site", default="mlp_up", choices=["mlp_up", "after_mlp", "cond_mlp"],
                    help="where the steering bias enters the drafter: mlp_up = Eq. 2 (SD^2), after_mlp = the "
                         "'Inv. Bias after MLP' ablation of Sec. 5, cond_mlp = its 'Cond. Bias in MLP' ablation")
    ap.add_argument("--pretrained", action="store_true",
                    help="the unsteered pretrained drafter (no steering stage, no bias): the baseline SD^2 "
                         "is compared with")
    ap.add_argument("--sweep", action="store_true",
                    help="instead of the iteration benchmark, the kernel sweep (one JSON line): acceptance "
                         "over vocab x batch x k, the steering step and Eq. 2 activation at both drafter widths "
                         "and four batch sizes, and the 8B-shaped verify at a 16384-token context")
    ap.add_argument("--sweep-parts", default="accept,steering,verify16k",
                    help="comma-separated parts of the kernel sweep to run (with --depth the 16K verify keeps "
                         "only the first layers: a profiling aid)")
    return ap.parse_args()


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except OSError:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0}, "fallback"


def workload_config(work, n_gpus, extra=None):
    cfg = {"workload": work.name + ": " + work.description, "batch_per_gpu": work.batch,
           "prompt_len": list(work.prompt_len), "k": work.k, "temperature": work.temperatures[-1],
           "gen_tokens": work.gen_tokens, "parallelism": f"replicas x{n_gpus}",
           "l2": "no flush: the weights streamed every step (%.1f GB) exceed the 126 MB L2" % (
               2e-9 * (work.verifier.param_count() + work.drafter.param_count()))
           if 2 * (work.verifier.param_count() + work.drafter.param_count()) > 126e6 else
           "weights fit in L2 (a parity-sized workload)"}
    if extra:
        cfg.update(extra)
    return cfg


# ---------------------------------------------------------------------------------------------
# clocks sampled during the timed region
# ---------------------------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except OSError:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for name, flag in zip(names, parts[5:9]):
                if flag.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------------------------
def timed_ms(fn, reps, flush):
    """Median device time of fn() over reps calls (CUDA events on the current stream), L2 flushed
    before each call outside the timed region, after two untimed calls."""
    for _ in range(2):
        fn()
    evs = []
    for _ in range(reps):
        flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        fn()
        e1.record()
        evs.append((e0, e1))
    torch.cuda.synchronize()
    return statistics.median(a.elapsed_time(b) for a, b in evs)


def run_sweep(args):
    """The kernel sweep on one GPU: acceptance (a4) over vocab {32000, 128256, 152064} x batch
    {1, 16, 64, 256} x k {1, 4, 8, 16} on bf16 logits N(0, 3^2) with a boosted token per row; the
    steering step (a1: g = LN(W_hml [h; m; l]), biases W_s g) and the Eq. 2 activation for the 2048-
    and 896-wide drafters at batch {1, 16, 64, 256} on random hidden states; the 8B-shaped verify
    stage at a 16384-token context, batch 1, k = 5, inside the captured iteration."""
    from paper_2511_09844_gb300 import build as _build
    from paper_2511_09844_gb300 import sd2
    _build.build()
    dev = "cuda:0"
    torch.cuda.set_device(0)
    peaks, _ = measured_peaks()
    hbm = float(peaks.get("hbm_gbs", 6800.0)) if peaks else 6800.0
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=dev)   # 256 MB > L2
    lib = sd2.load_library()
    out = {"mode": "kernel sweep", "timing": "median of CUDA-event times per call, L2 flushed before each call",
           "peak_hbm_gbs": hbm}
    parts = set(args.sweep_parts.split(","))

    acc = []
    for V in ((32000, 128256, 152064) if "accept" in parts else ()):
        for B in (1, 16, 64, 256):
            for k in (1, 4, 8, 16):
                target, draft, xhat = W.make_sweep_logits(B, k, V, seed=11, device=dev)
                temp = torch.ones(B, dtype=torch.float32, device=dev)
                ws = torch.empty(lib.sd2_accept_workspace_bytes(B, k), dtype=torch.uint8, device=dev)
                step = [0]

                def call():
                    step[0] += 1
                    sd2.accept_logits(target, draft, xhat, temp, seed=5, step=step[0], workspace=ws)
                ms = timed_ms(call, 10, flush)
                nbytes = (target.numel() + draft.numel()) * 2      # every logit read once: (2k+1) V B bf16
                acc.append({"V": V, "B": B, "k": k, "ms": round(ms, 4), "logit_bytes": nbytes,
                            "gbs": round(nbytes / (ms / 1e3) / 1e9, 1)})
                del target, draft, xhat, ws
    if acc:
        out["accept"] = acc

    steer = []
    for name in (("llama8b_1b", "qwen32b_05b") if "steering" in parts else ()):
        work = W.WORKLOADS[name]
        st = W.make_steering_weights(work, 21, device=dev)
        dv, dg, F = work.verifier.d_model, work.d_steer, work.bias_width
        n_bias = work.drafter.n_layers * F
        wbytes = (st["w_hml"].numel() + st["w_s"].numel()) * 2
        for B in (1, 16, 64, 256):
            g = torch.Generator(device=dev).manual_seed(B)
            taps = torch.randn(B, 3, dv, generator=g, device=dev)
            ms = timed_ms(lambda: sd2.steer(taps, st, work.steer_ln_eps, n_bias), 10, flush)
            nbytes = wbytes + taps.numel() * 4 + B * (dg + n_bias) * 4
            gate = torch.randn(B, F, generator=g, device=dev)
            up = torch.randn(B, F, generator=g, device=dev)
            bias = torch.randn(B, F, generator=g, device=dev)
            seq = torch.arange(B, dtype=torch.int32, device=dev)
            ms2 = timed_ms(lambda: sd2.swiglu_steered(gate, up, bias, seq), 10, flush)
            steer.append({"pair": name, "d_v": dv, "d_g": dg, "d_d": work.drafter.d_model, "F_D": F, "B": B,
                          "steer_ms": round(ms, 4), "steer_bytes": nbytes,
                          "steer_gbs": round(nbytes / (ms / 1e3) / 1e9, 1),
                          "eq2_ms": round(ms2, 4), "eq2_bytes": B * F * 14})
        del st
    if steer:
        out["steering"] = steer
    if "verify16k" not in parts:
        return out

    # the verify stage at a 16384-token context (batch 1, k = 5) inside the captured iteration
    work = bench_workload(argparse.Namespace(workload="llama8b_1b", steer_site="mlp_up", depth=args.depth))
    prompts = W.make_prompts(work.verifier.vocab, 1, (16384, 16384), seed=7)
    vw, dw, st = make_device_weights(work, args.seed, dev)
    eng = sd2.SD2Engine(work, vw, dw, st, max_batch=1, max_ctx=16384 + 40 * (work.k + 1),
                        max_prefill_tokens=16384, stream=torch.cuda.current_stream())
    eng.prefill(prompts, [1.0], seed=args.seed)
    for _ in range(4):
        eng.step()
        eng.accept()
    eng.stage_timing(True)
    st_ms = {"steer": 0.0, "draft": 0.0, "verify": 0.0}
    for _ in range(8):
        eng.step()
        eng.accept()
        for key, v in eng.stage_read().items():
            st_ms[key] += v / 8
    eng.stage_timing(False)
    v = work.verifier
    ctx = 16384 + 8 * (work.k + 1) // 2             # about the mean context of the timed steps
    kv = ctx * v.n_layers * 2 * v.n_kv_heads * v.head_dim * 2
    per_layer = v.d_model * (v.n_heads + 2 * v.n_kv_heads) * v.head_dim + v.n_heads * v.head_dim * v.d_model \
        + 3 * v.d_ffn * v.d_model
    wts = (v.n_layers * per_layer + v.vocab * v.d_model) * 2   # every non-embedding weight incl. lm_head, bf16
    ms = st_ms["verify"]
    out["verify_16k"] = {"context": 16384, "B": 1, "k": work.k, "verify_layers": v.n_layers,
                         "verify_ms": round(ms, 4),
                         "weight_bytes": wts, "kv_read_bytes": kv,
                         "gbs": round((wts + kv) / (ms / 1e3) / 1e9, 1),
                         "frac_of_measured_hbm": round((wts + kv) / (ms / 1e3) / 1e9 / hbm, 4),
                         "draft_step_ms": round(st_ms["draft"] / work.k, 4),
                         "timing": "CUDA event nodes between the stages of the captured iteration, mean of 8"}
    return out


def sm_count_of(dev):
    return torch.cuda.get_device_properties(dev).multi_processor_count


def gemm_traffic(algorithmic_bytes_per_launch):
    """DRAM bytes per GEMM launch from the committed ncu record, if it was taken on this source."""
    import hashlib
    rec_path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "profiles", "gemm_tc_traffic.json")
    try:
        rec = json.load(open(rec_path))
        src = os.path.join(os.path.dirname(os.path.abspath(__file__)), rec["source"])
        if hashlib.sha256(open(src, "rb").read()).hexdigest() != rec["source_sha256"]:
            return None
        return round(algorithmic_bytes_per_launch * float(rec["dram_bytes_per_algorithmic_byte"]))
    except (OSError, KeyError, ValueError):
        return None


def bench_workload(args):
    """The named workload; with --depth, its models cut to their first layers (profiling aid)."""
    import dataclasses
    work = W.WORKLOADS[args.workload]
    if args.steer_site != work.steering_site:
        work = dataclasses.replace(work, steering_site=args.steer_site)
    if args.depth:
        lv, ld = (int(x) for x in args.depth.split(","))
        work = dataclasses.replace(work, verifier=dataclasses.replace(work.verifier, n_layers=lv),
                                   drafter=dataclasses.replace(work.drafter, n_layers=ld))
    return work


def make_device_weights(work, seed, device):
    vw = W.make_lm_weights(work.verifier, seed, device=device)
    dw = W.make_lm_weights(work.drafter, seed + 1, device=device)
    st = W.make_steering_weights(work, seed + 2, device=device)
    return vw, dw, st


def gemm_stamp_summary(steps, hbm):
    """The weight-streaming GEMM's roofline from the in-graph globaltimer stamps of several steps.

    Each launch's time is its exposed duration: from the later of its programmatic wait returning
    (the kernel before it has completed) and the previous GEMM's exit, to its own exit. These
    intervals do not overlap and lie inside the step, so their sum is at most the step's time;
    weight bytes a kernel prefetched before its wait count for it, the wait itself does not."""
    tot_ns, tot_bytes, n = 0, 0.0, 0
    by_stage = {"steer": [0, 0.0], "draft": [0, 0.0], "verify": [0, 0.0]}
    span = 0
    for launches in steps:
        prev_exit = None
        k1 = max(l["stage"] for l in launches)
        for l in launches:
            start = l["wait"] if prev_exit is None else max(l["wait"], prev_exit)
            dur = max(0, l["exit"] - start)
            prev_exit = l["exit"] if prev_exit is None else max(prev_exit, l["exit"])
            tot_ns += dur
            tot_bytes += l["bytes"]
            n += 1
            key = "steer" if l["stage"] == 0 else ("verify" if l["stage"] == k1 else "draft")
            by_stage[key][0] += dur
            by_stage[key][1] += l["bytes"]
        span += launches[-1]["exit"] - min(l["entry"] for l in launches)
    ns = len(steps)
    gbs = tot_bytes / (tot_ns * 1e-9) / 1e9 if tot_ns else 0.0
    out = {"achieved": round(gbs, 1), "frac": round(gbs / hbm, 4), "gemm_ms_per_step": round(tot_ns / ns / 1e6, 4),
           "launches_per_step": n // ns, "bytes_per_launch": round(tot_bytes / n),
           "avg_launch_us": round(tot_ns / n / 1e3, 3), "gemm_span_ms_per_step": round(span / ns / 1e6, 4)}
    for key, (t, b) in by_stage.items():
        if t:
            out[f"{key}_gbs"] = round(b / (t * 1e-9) / 1e9, 1)
            out[f"{key}_frac"] = round(b / (t * 1e-9) / 1e9 / hbm, 4)
    return out


def committed_len(eng):
    """Committed length of each sequence (host read of the device state; outside timed regions)."""
    st = eng.buffer(7)
    return st[:eng.batch].tolist()


def timed_steps(eng, steps, stream):
    """K graph-replayed iterations bracketed by CUDA events on the engine's stream: (ms, emitted)."""
    B, k = eng.batch, eng.k
    n_all = torch.zeros((steps, B), dtype=torch.int32, device="cuda")
    tok_all = torch.zeros((steps, B, k + 1), dtype=torch.int32, device="cuda")
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    ev0.record(stream)
    for i in range(steps):
        eng.step()
        eng.accept(tok_all[i], n_all[i])
    ev1.record(stream)
    torch.cuda.synchronize()
    return ev0.elapsed_time(ev1), int(n_all.sum().item())


def stage_times(eng, steps):
    eng.stage_timing(True)
    acc = {"steer": 0.0, "draft": 0.0, "verify": 0.0}
    for _ in range(steps):
        eng.step()
        eng.accept()
        for key, v in eng.stage_read().items():
            acc[key] += v / steps
    eng.stage_timing(False)
    return acc


def stage_bytes(work):
    """Weights streamed by one verify (a3) and by one drafter step (a2): every layer + lm_head."""
    def model(m):
        per = m.d_model * (m.n_heads + 2 * m.n_kv_heads) * m.head_dim + m.n_heads * m.head_dim * m.d_model \
            + 3 * m.d_ffn * m.d_model
        return 2.0 * (m.n_layers * per + m.vocab * m.d_model)
    return model(work.verifier), model(work.drafter)


def advance_to(eng, target):
    """Untimed iterations until every sequence's committed length reaches `target`: the timed
    steps then sit in the middle of the configuration's generation instead of right after the prompt."""
    steps = 0
    while min(committed_len(eng)) < target and steps < 10000:
        eng.step()
        eng.accept()
        steps += 1
    return steps


def run_ours(args, rank, world, local_rank):
    from paper_2511_09844_gb300 import build as _build
    from paper_2511_09844_gb300 import sd2
    _build.build()
    torch.cuda.set_device(local_rank)
    dev = f"cuda:{local_rank}"
    work = bench_workload(args)
    B, k, V = work.batch, work.k, work.verifier.vocab
    temp = work.temperatures[-1]
    prompts = W.make_prompts(V, B, work.prompt_len, seed=7 + rank)
    plen = max(len(p) for p in prompts)
    # the timed steps start at about prompt + gen/2 - steps tokens, i.e. around the middle of the
    # configuration's generation (tau ~ 2 tokens per step)
    start_ctx = plen + work.gen_tokens // 2 - args.steps
    max_ctx = plen + work.gen_tokens + (args.warmup + args.steps + 16) * (k + 1) + k + 8
    vw, dw, st = make_device_weights(work, args.seed, dev)
    stream = torch.cuda.current_stream()
    peaks, peak_src = measured_peaks()
    hbm = float(peaks["hbm_gbs"])
    eng = sd2.SD2Engine(work, vw, dw, st, max_batch=B, max_ctx=max_ctx,
                        max_prefill_tokens=sum(len(p) for p in prompts), stream=stream,
                        steering=not args.pretrained)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    eng.prefill(prompts, [temp] * B, seed=args.seed + rank)
    torch.cuda.synchronize()
    prefill_s = time.perf_counter() - t0
    advance = advance_to(eng, start_ctx)
    for _ in range(args.warmup):
        eng.step()
        eng.accept()
    torch.cuda.synchronize()
    ctx0 = committed_len(eng)
    barrier(world)
    with ClockSampler(local_rank) as clocks:
        ms, emitted = timed_steps(eng, args.steps, stream)
    barrier(world)
    ctx1 = committed_len(eng)
    ms_max, emitted_all = reduce_max_sum(ms, emitted, world)
    value = emitted_all / B / (ms_max / 1e3)
    tau = emitted / (args.steps * B)

    # stage times inside the captured step (event nodes between the stages)
    stage_steps = min(args.steps, 8)
    st_ms = stage_times(eng, stage_steps)
    verify_bytes, draft_bytes = stage_bytes(work)
    verify_gbs = verify_bytes / (st_ms["verify"] / 1e3) / 1e9 if st_ms["verify"] else 0.0
    draft_gbs = draft_bytes / (st_ms["draft"] / k / 1e3) / 1e9 if st_ms["draft"] else 0.0

    # the GEMM's roofline from globaltimer stamps inside the captured step
    eng.gemm_timing(True)
    stamped = []
    for _ in range(stage_steps):
        eng.step()
        eng.accept()
        stamped.append(eng.gemm_timing_read())
    eng.gemm_timing(False)
    gemm = gemm_stamp_summary(stamped, hbm)

    # kernel launches per iteration: one pass with the per-launch profile (no graphs, not timed)
    eng.profile(True)
    for _ in range(2):
        eng.step()
        eng.accept()
    prof = eng.profile_read()
    eng.profile(False)
    launches_per_step = sum(v["launches"] for name, v in prof.items()
                            if name in ("gemm", "attention", "accept", "sample", "other")) / 2
    eng.check()

    # end to end through the public API on host buffers: one whole request of the configuration
    # (prompt upload, prefill, decode until gen_tokens new tokens per sequence, every step's
    # tokens copied back to host memory), host wall clock
    e2e_runs = []
    for r in range(3):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        out = eng.generate(prompts, [temp] * B, seed=args.seed + rank + 100 * r, max_new=work.gen_tokens)
        e2e_runs.append((time.perf_counter() - t0, sum(len(o) for o in out)))
    e2e_s = statistics.median(t for t, _ in e2e_runs)
    e2e_tokens = e2e_runs[0][1]
    e2e_s_max, e2e_all = reduce_max_sum(e2e_s * 1e3, e2e_tokens, world)
    e2e_value = e2e_all / B / (e2e_s_max / 1e3)
    e2e_steps = max(1, round((e2e_tokens / B - 1) / max(tau, 1e-9)))
    h2d_req = 4 * sum(len(p) for p in prompts) + 4 * B
    eng.close()
    keep = (vw, dw, st) if (rank == 0 and world == 1 and not args.no_cpu_baseline) else None
    extras = None
    if not args.depth and not args.no_extras and rank == 0:
        extras = other_workloads(sd2, dev, args, hbm, vw, dw, st)
    del vw, dw, st

    line = {
        "metric": METRIC, "value": round(value, 3), "unit": "tokens/s/sequence", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_max / args.steps, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic: random-init bf16 weights N(0, 0.02^2), uniform-random prompt ids",
        "config": workload_config(work, world, dict(**({"depth": f"{work.verifier.n_layers} verifier + "
                                                                  f"{work.drafter.n_layers} drafter layers "
                                                                  "(profiling aid, not the workload)"}
                                                        if args.depth else {}),
                                                    **({"drafter": "pretrained, unsteered (no steering stage)"}
                                                       if args.pretrained else {}),
                                                    **({"steering_site": {"after_mlp": "after the MLP (Sec. 5 ablation)",
                                                                          "cond_mlp": "conditional bias MLP (Sec. 5 ablation)"}
                                                        [work.steering_site]}
                                                       if work.steering_site != "mlp_up" else {}))),
        "timed_context": {"start": ctx0, "end": ctx1, "untimed_steps_before": advance + args.warmup,
                          "note": "the timed steps sit around the middle of the configuration's generation "
                                  "(prompt + gen_tokens/2); e2e runs whole requests of gen_tokens"},
        "max_ctx": max_ctx,
        "tau": round(tau, 4),
        "tokens_per_s_at_paper_tau": {"tau": 5.00, "value": round(5.00 / (ms_max / args.steps / 1e3), 2)},
        "prefill_s": round(prefill_s, 3),
        "e2e": {"value": round(e2e_value, 3), "unit": "tokens/s/sequence",
                "h2d_bytes_per_step": int(round(h2d_req / e2e_steps)),
                "d2h_bytes_per_step": 4 * B * (k + 2),
                "h2d_bytes_per_request": h2d_req, "new_tokens_per_sequence": work.gen_tokens,
                "seconds_per_request": [round(t, 4) for t, _ in e2e_runs],
                "how": "sd2_generate (C ABI, host buffers): prompt upload, prefill, sd2_step + sd2_accept until "
                       f"{work.gen_tokens} new tokens per sequence, each step's tokens copied to host and waited "
                       "for; host wall clock, median of 3 requests (the step graphs are captured during the first and "
                       "reused by the later ones: a new prefill of the same batch size keeps them)"},
        "roofline": dict({"bound": "hbm", "kernel": "weight-streaming GEMM (gemm_tc_kernel: all projections + lm_head)",
                          "peak": hbm, "unit": "GB/s",
                          "traffic": gemm_traffic(gemm["bytes_per_launch"]),
                          "traffic_note": "DRAM bytes per launch: the algorithmic bytes per launch x the "
                                          "DRAM/algorithmic ratio ncu measured on this kernel source "
                                          "(profiles/gemm_tc_traffic.json); null if the source changed since",
                          "peak_source": f"{peak_src} hbm_gbs (MEASURED_PEAKS.json)" if peak_src == "measured" else
                          "fallback 6800 GB/s",
                          "timing": f"globaltimer stamps of every GEMM launch inside the captured step, {stage_steps} "
                                    "steps: per launch from its programmatic wait returning (or the previous GEMM's "
                                    "exit, if later) to its last CTA's exit; achieved = algorithmic bytes / that time"},
                         **gemm),
        "stages": {"timing": f"CUDA event nodes between the stages of the captured step, mean of {stage_steps} steps",
                   "bytes": "weights streamed per stage (verify: all layers + lm_head; draft step: all layers + lm_head)",
                   "verify_ms": round(st_ms["verify"], 4), "verify_gb": round(verify_bytes / 1e9, 3),
                   "verify_gbs": round(verify_gbs, 1), "verify_frac_of_8tbs": round(verify_gbs / NOMINAL_HBM_GBS, 4),
                   "verify_frac_of_measured": round(verify_gbs / hbm, 4),
                   "draft_step_ms": round(st_ms["draft"] / k, 4), "draft_step_gb": round(draft_bytes / 1e9, 3),
                   "draft_step_gbs": round(draft_gbs, 1), "draft_step_frac_of_measured": round(draft_gbs / hbm, 4),
                   "steer_ms": round(st_ms["steer"], 4)},
        "gpu_launches": int(round(launches_per_step * args.steps)),
        "clocks": clocks.summary(),
    }
    if extras:
        line["other_configs"] = extras
    return line, work, tau, keep


def run_pair(sd2, work, vw, dw, st, hbm, steps=10, warmup=3, max_ctx=None, temps=None, seed=1234):
    """One workload's iteration in the captured graph: ms, tau, emitted tokens/s/seq, stage fractions."""
    B, k, V = work.batch, work.k, work.verifier.vocab
    prompts = W.make_prompts(V, B, work.prompt_len, seed=7)
    temps = temps or [work.temperatures[b % len(work.temperatures)] for b in range(B)]
    plen = max(len(p) for p in prompts)
    max_ctx = max_ctx or plen + (warmup + steps + 8 + 8) * (k + 1) + k + 8
    eng = sd2.SD2Engine(work, vw, dw, st, max_batch=B, max_ctx=max_ctx, max_prefill_tokens=sum(len(p) for p in prompts),
                        stream=torch.cuda.current_stream())
    eng.prefill(prompts, temps, seed=seed)
    for _ in range(warmup):
        eng.step()
        eng.accept()
    ms, emitted = timed_steps(eng, steps, torch.cuda.current_stream())
    sms = stage_times(eng, 4)
    eng.check()
    eng.close()
    vb, db = stage_bytes(work)
    it = ms / steps
    return {"ms_per_iteration": round(it, 4), "tau": round(emitted / (steps * B), 4),
            "tokens_per_s_per_sequence": round(emitted / B / (ms / 1e3), 2),
            "verify_ms": round(sms["verify"], 4), "verify_frac_of_measured": round(vb / (sms["verify"] / 1e3) / 1e9 / hbm, 4),
            "draft_step_ms": round(sms["draft"] / k, 4),
            "draft_step_frac_of_measured": round(db / (sms["draft"] / k / 1e3) / 1e9 / hbm, 4),
            "steer_ms": round(sms["steer"], 4)}


def other_workloads(sd2, dev, args, hbm, vw8, dw1, st8):
    """The other configurations, each timed in the captured graph on its own workload: the 8B/1B pair
    at batch 16 (ragged prompts, k = 8, T in {0, 0.7, 1}), the Qwen-32B/0.5B pair (batch 4, prompt
    2048, k = 6), and the kernel sweep's corners (acceptance, steering) and its 16K-context verify."""
    out = {}
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=dev)   # 256 MB > L2
    b16 = W.WORKLOADS["llama8b_1b_b16"]
    out["llama8b_1b_b16"] = dict({"config": b16.description}, **run_pair(sd2, b16, vw8, dw1, st8, hbm))
    # the 16K-context verify of the kernel sweep (8B-shaped, batch 1, k = 5)
    w8 = W.WORKLOADS["llama8b_1b"]
    prompts = W.make_prompts(w8.verifier.vocab, 1, (16384, 16384), seed=7)
    eng = sd2.SD2Engine(w8, vw8, dw1, st8, max_batch=1, max_ctx=16384 + 40 * (w8.k + 1), max_prefill_tokens=16384,
                        stream=torch.cuda.current_stream())
    eng.prefill(prompts, [1.0], seed=args.seed)
    for _ in range(4):
        eng.step()
        eng.accept()
    sms = stage_times(eng, 8)
    eng.check()
    eng.close()
    v = w8.verifier
    kv = (16384 + 8) * v.n_layers * 2 * v.n_kv_heads * v.head_dim * 2
    vb, _ = stage_bytes(w8)
    out["verify_16k"] = {"config": "8B-shaped verify at context 16384, batch 1, k = 5 (kernel sweep)",
                         "verify_ms": round(sms["verify"], 4), "weight_bytes": vb, "kv_read_bytes": kv,
                         "frac_of_measured": round((vb + kv) / (sms["verify"] / 1e3) / 1e9 / hbm, 4),
                         "draft_step_ms": round(sms["draft"] / w8.k, 4)}
    # acceptance corners (bf16 logits N(0, 3^2) with a boosted token per row, V = 152064)
    lib = sd2.load_library()
    acc = []
    for B, k in ((1, 1), (1, 16), (256, 1), (256, 16)):
        V = 152064
        target, draft, xhat = W.make_sweep_logits(B, k, V, seed=11, device=dev)
        temp = torch.ones(B, dtype=torch.float32, device=dev)
        ws = torch.empty(lib.sd2_accept_workspace_bytes(B, k), dtype=torch.uint8, device=dev)
        step = [0]

        def call():
            step[0] += 1
            sd2.accept_logits(target, draft, xhat, temp, seed=5, step=step[0], workspace=ws)
        ms = timed_ms(call, 10, flush)
        nbytes = (target.numel() + draft.numel()) * 2
        acc.append({"V": V, "B": B, "k": k, "ms": round(ms, 4), "logit_bytes": nbytes,
                    "frac_of_measured_hbm_one_read": round(nbytes / (ms / 1e3) / 1e9 / hbm, 4)})
        del target, draft, xhat, ws
    out["accept_corners"] = {"config": "sd2_accept_logits, bf16 logits N(0, 3^2) + one boosted token per row, "
                                       "L2 flushed before each call, median of 10", "points": acc}
    # steering step at both drafter widths
    steer = []
    for name in ("llama8b_1b", "qwen32b_05b"):
        wk = W.WORKLOADS[name]
        stw = W.make_steering_weights(wk, 21, device=dev)
        dv, dg, F = wk.verifier.d_model, wk.d_steer, wk.bias_width
        n_bias = wk.drafter.n_layers * F
        wbytes = (stw["w_hml"].numel() + stw["w_s"].numel()) * 2
        for B in (1, 256):
            taps = torch.randn(B, 3, dv, generator=torch.Generator(device=dev).manual_seed(B), device=dev)
            ms = timed_ms(lambda: sd2.steer(taps, stw, wk.steer_ln_eps, n_bias), 10, flush)
            nbytes = wbytes + taps.numel() * 4 + B * (dg + n_bias) * 4
            steer.append({"pair": name, "d_d": wk.drafter.d_model, "B": B, "ms": round(ms, 4),
                          "frac_of_measured_hbm": round(nbytes / (ms / 1e3) / 1e9 / hbm, 4)})
        del stw
    out["steering"] = {"config": "sd2_steer on random hidden states N(0,1), L2 flushed, median of 10", "points": steer}
    del flush
    # the Qwen-32B / 0.5B pair
    q = W.WORKLOADS["qwen32b_05b"]
    qv, qd, qs = make_device_weights(q, args.seed, dev)
    out["qwen32b_05b"] = dict({"config": q.description}, **run_pair(sd2, q, qv, qd, qs, hbm))
    del qv, qd, qs
    torch.cuda.empty_cache()
    return out


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def reduce_max_sum(ms, count, world):
    """(max of ms over the ranks, sum of count over the ranks): the job's time is its slowest
    replica's, its work every replica's."""
    if world == 1:
        return ms, count
    import torch.distributed as dist
    device = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    c = torch.tensor([count], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(c, op=dist.ReduceOp.SUM)
    return float(t.item()), int(c.item())


# ---------------------------------------------------------------------------------------------
# the oracle on the host cores (reference arm and cpu_baseline)
# ---------------------------------------------------------------------------------------------
class OracleSlices:
    """The oracle on two slices of the workload (1 and 2 decoder layers per model, same widths,
    same context); the difference prices one layer, which scales the slice to the full depth.
    Weights: the first layers of the given models (copied to the host), or freshly generated.
    The context is the prompt plus half the configuration's generation, where the GPU arm's
    timed steps sit. Each repeat draws its random numbers from its own seed, so the accepted
    drafts of the repeats sample the oracle's own block efficiency tau on the slices."""

    def __init__(self, work, seed, weights=None):
        import dataclasses
        self.work = work
        self.context = work.prompt_len[0] + work.gen_tokens // 2
        two_v = dataclasses.replace(work.verifier, n_layers=2)
        two_d = dataclasses.replace(work.drafter, n_layers=2)
        if weights is None:
            sw2 = dataclasses.replace(work, verifier=two_v, drafter=two_d)
            vw, dw, st = (W.make_lm_weights(two_v, seed), W.make_lm_weights(two_d, seed + 1),
                          W.make_steering_weights(sw2, seed + 2))
        else:
            vw, dw, st = weights

        def host(w, n):
            return {"embed": w["embed"].cpu(), "final_norm": w["final_norm"].cpu(), "lm_head": w["lm_head"].cpu(),
                    "layers": [{k: v.cpu() for k, v in lw.items()} for lw in w["layers"][:n]]}

        vh, dh = host(vw, 2), host(dw, 2)
        F = work.drafter.d_ffn
        sth = {k: v.cpu() for k, v in st.items()}
        self.slices = []
        for n in (1, 2):
            vs = dataclasses.replace(work.verifier, n_layers=n)
            ds = dataclasses.replace(work.drafter, n_layers=n)
            sw = dataclasses.replace(work, verifier=vs, drafter=ds)
            v_n = dict(vh, layers=vh["layers"][:n])
            d_n = dict(dh, layers=dh["layers"][:n])
            st_n = dict(sth, w_s=sth["w_s"][:n * F])
            self.slices.append((sw, v_n, d_n, st_n))
        self.prompt = W.make_prompts(work.verifier.vocab, 1, (self.context, self.context), seed=7)[0]
        self.seed = seed
        self.blocks = []          # tokens emitted per oracle iteration (j + 1)

    def _iteration(self, sl, rep):
        from oracle.sd import OracleSD
        sw, vw, dw, st = sl
        ora = OracleSD(sw, vw, dw, st, self.seed + rep)
        ora.prefill([self.prompt], [self.work.temperatures[-1]], forced_first=[1])
        t0 = time.perf_counter()
        out = ora.stage(0, 1)
        emitted, j = ora.accept(0, 1, out)
        ora.commit(0, emitted, j, out["taps"])
        self.blocks.append(j + 1)
        return time.perf_counter() - t0

    def estimate(self, rep=0):
        """(seconds per iteration scaled to full depth, seconds of CPU work measured)."""
        t1 = self._iteration(self.slices[0], rep)
        t2 = self._iteration(self.slices[1], rep)
        per_pair = max(0.0, t2 - t1)                       # one verifier layer + one drafter layer (x k)
        fixed = max(0.0, t1 - per_pair)
        work = self.work
        vcost = work.verifier.param_count() / work.verifier.n_layers
        dcost = work.k * work.drafter.param_count() / work.drafter.n_layers
        v_share = vcost / (vcost + dcost)
        full = fixed + per_pair * (v_share * work.verifier.n_layers + (1 - v_share) * work.drafter.n_layers)
        return full, t1 + t2

    def tau(self):
        return statistics.mean(self.blocks) if self.blocks else 1.0

    def sample_text(self, measured):
        w = self.work
        return (f"oracle iterations (fp32, full recompute, no KV cache) on 1- and 2-layer slices of the "
                f"same shapes at context {self.context}, scaled to {w.verifier.n_layers} verifier + "
                f"{w.drafter.n_layers} drafter layers (per-iteration seconds extrapolated from the two "
                f"slices, not a full-depth run); {round(measured, 1)} s of CPU work; tau {round(self.tau(), 3)} "
                f"= the oracle's own mean emitted tokens per iteration over {len(self.blocks)} iterations")


def run_reference(args, rank, world):
    if rank != 0:
        return None
    work = W.WORKLOADS[args.workload]
    sl = OracleSlices(work, args.seed)
    for r in range(args.warmup):
        sl.estimate(rep=r)
    sl.blocks.clear()
    per_step, cpu_s = [], 0.0
    t_start = time.perf_counter()
    for r in range(args.steps):
        est, measured = sl.estimate(rep=args.warmup + r)
        per_step.append(est)
        cpu_s += measured
        if time.perf_counter() - t_start > 150:      # keep the arm within a few minutes
            break
    t_iter = statistics.median(per_step)
    tau = sl.tau()
    value = tau / t_iter
    return {
        "impl": "reference", "metric": METRIC, "value": round(value, 6), "unit": "tokens/s/sequence",
        "n_gpus": world, "steps": len(per_step), "warmup": args.warmup, "ms_per_step": round(t_iter * 1e3, 2),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic: random-init bf16 weights N(0, 0.02^2), uniform-random prompt ids",
        "config": workload_config(work, 1),
        "tau": round(tau, 4), "seconds_per_iteration": round(t_iter, 3),
        "cpu_baseline": {"value": round(value, 6), "unit": "tokens/s/sequence", "cores": torch.get_num_threads(),
                         "kind": "oracle", "sample": sl.sample_text(cpu_s)},
        "e2e": {"value": round(value, 6), "unit": "tokens/s/sequence", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }


def cpu_baseline(work, seed, weights=None, min_cpu_s=10.0, max_repeats=8):
    """The oracle's sliced iteration, repeated (each with its own seed) until about min_cpu_s of
    CPU work is measured; the median of the scaled estimates, at the oracle's own tau. Then one
    more estimate on a single thread."""
    sl = OracleSlices(work, seed, weights)
    ests, measured = [], 0.0
    while measured < min_cpu_s and len(ests) < max_repeats:
        est, m = sl.estimate(rep=len(ests))
        ests.append(est)
        measured += m
    est = statistics.median(ests)
    tau = sl.tau()
    out = {"value": round(tau / est, 6), "unit": "tokens/s/sequence", "cores": torch.get_num_threads(),
           "kind": "oracle", "seconds_per_iteration": round(est, 3), "repeats": len(ests), "tau": round(tau, 4),
           "sample": sl.sample_text(measured) + f"; median of {len(ests)} repeats"}
    threads = torch.get_num_threads()
    torch.set_num_threads(1)
    try:
        est1, m1 = sl.estimate(rep=len(ests))
    finally:
        torch.set_num_threads(threads)
    out["single_thread"] = {"value": round(tau / est1, 6), "seconds_per_iteration": round(est1, 3), "cores": 1,
                            "cpu_seconds": round(m1, 1)}
    return out


def main():
    args = parse()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if args.impl == "ours" else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local_rank)
        dist.init_process_group(backend)
    if args.sweep:
        line = run_sweep(args) if rank == 0 else None
    elif args.impl == "reference":
        line = run_reference(args, rank, world)
    else:
        line, work, tau, keep = run_ours(args, rank, world, local_rank)
        if keep is not None:
            line["cpu_baseline"] = cpu_baseline(work, args.seed, keep)
    if rank == 0 and line is not None:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
