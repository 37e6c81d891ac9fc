"""Benchmark of the Jacobi-decoding hot path on GB300: committed tokens/s on the Qwen2.5-7B-shaped
bf16 decoder at batch 1 (prompt 1024, block n = 32, 512 new tokens, draft injection p = 0.3
against the model's own greedy continuation, paged KV with 16-token pages).

One step = one jf_generate_device call: prefill of the prompt plus every Jacobi iteration until
512 new tokens are committed. Inputs are resident on the device when the timed region starts
(`value`); `e2e` repeats the measurement through jf_generate with host buffers (prompt and truth
copied in, tokens copied out inside the timed region).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference] [--no-cpu-baseline]

For N > 1 (torchrun) every rank runs an independent replica of the workload (the path does not
shard); value = tokens of all ranks / max-over-ranks time.
"""
from __future__ import annotations

import argparse
import dataclasses
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "tokens/s at bs1 on 7B-shape; Jacobi-iteration latency as % of HBM roofline"
NOMINAL_HBM_GBS = 8000.0


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    shape: str          # key of paper_2512_14681_gb300.inputs.SHAPES
    prompt: int
    block: int          # n
    new: int
    p: float            # draft-injection corruption rate
    blocks: int = 1     # K (multi-block decoding)
    pool: int = 0       # rejection-recycling pool entries
    ngram: int = 0      # n-gram length (0 = n)
    cands: int = 0      # recycled candidates verified per iteration
    spawn: float = 0.0  # spawn ratio r: a new block starts once the newest has ceil(r n) accepted tokens


# The 7B single-block workload at p = 0.3 is the headline; the others are the remaining decode
# configurations of the same family (1.5B single block; 7B at p = 0.1 / 0.7; 7B multi-block with
# rejection recycling). Prompts are uniform-random tokens, weights N(0, 0.02).
WORKLOADS = {w.name: w for w in [
    Workload("qwen2.5-7b-shape-bf16 prompt1024 block32 new512 inject-p0.3 paged-kv16 bs1",
             "qwen2.5-7b-shape-bf16", 1024, 32, 512, 0.3),
    Workload("qwen2.5-7b-shape-bf16 prompt1024 block32 new512 inject-p0.1 paged-kv16 bs1",
             "qwen2.5-7b-shape-bf16", 1024, 32, 512, 0.1),
    Workload("qwen2.5-7b-shape-bf16 prompt1024 block32 new512 inject-p0.7 paged-kv16 bs1",
             "qwen2.5-7b-shape-bf16", 1024, 32, 512, 0.7),
    Workload("qwen2.5-1.5b-shape-bf16 prompt512 block16 new256 inject-p0.5 paged-kv16 bs1",
             "qwen2.5-1.5b-shape-bf16", 512, 16, 256, 0.5),
    Workload("qwen2.5-7b-shape-bf16 prompt2048 blocks4x32 rr-pool64x32 cand1 new1024 inject-p0.3 paged-kv16 bs1",
             "qwen2.5-7b-shape-bf16", 2048, 32, 1024, 0.3, blocks=4, pool=64, ngram=32, cands=1),
    # the paper's inference configuration for its method (Sec. 4.3 / App. E): K = 2 blocks of n = 64,
    # spawn ratio r = 0.85, 4 recycled n-grams verified per iteration (up to 384 rows in flight)
    Workload("qwen2.5-7b-shape-bf16 prompt1024 blocks2x64 spawn0.85 rr-pool64x64 cand4 new512 inject-p0.3 paged-kv16 bs1",
             "qwen2.5-7b-shape-bf16", 1024, 64, 512, 0.3, blocks=2, pool=64, ngram=64, cands=4, spawn=0.85),
]}
DEFAULT_WORKLOAD = next(iter(WORKLOADS))
ALIASES = {"7b": DEFAULT_WORKLOAD, "7b-p0.1": list(WORKLOADS)[1], "7b-p0.7": list(WORKLOADS)[2],
           "1.5b": list(WORKLOADS)[3], "7b-mb4-rr": list(WORKLOADS)[4], "7b-mr-k2n64": list(WORKLOADS)[5]}
# DRAM bytes (read + write) per launch of the gate/up projection at M = 32 rows: dram__bytes_read.sum
# + dram__bytes_write.sum of one `ncu --set full` capture of the current kernel (271.87 MB weights
# and activations read, 3.49 MB SwiGLU output written). Set to None whenever the kernel changes.
GATEUP_TRAFFIC_BYTES = 275_357_696


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi clocks/throttle reasons sampled during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.dev = device_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "200",
                 "-i", str(self.dev)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.t.join(timeout=2)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [x.strip() for x in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower() in ("active", "1", "0x1"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def aggregate_ranks(local_ms: float, local_tokens: int, dist=None, device=None):
    """Whole-job throughput of independent replicas: every rank's tokens over the slowest rank's
    time (max over ranks of the timed region). Returns (max_ms, total_tokens, tokens_per_s)."""
    import torch

    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return local_ms, local_tokens, local_tokens / (local_ms / 1000.0)
    t = torch.tensor([local_ms], dtype=torch.float64, device=device)
    n = torch.tensor([float(local_tokens)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(n, op=dist.ReduceOp.SUM)
    max_ms, total = float(t.item()), int(n.item())
    return max_ms, total, total / (max_ms / 1000.0)


# ------------------------------------------------------------------------------------------
# CPU oracle sample (the reference arm and the cpu_baseline object)
# ------------------------------------------------------------------------------------------
def oracle_sample(steps: int, warmup: int, prompt_len: int = 16):
    """Per-iteration figure of the oracle (fp64 C, OpenMP over the machine's host cores) on the headline
    workload's model and decoding parameters: the 7B-shaped bf16 model, block n = 32, drafts injected
    at p = 0.3 against the oracle's own greedy continuation. The oracle prefills the first
    `prompt_len` prompt tokens (a 1,024-token prefill alone takes minutes on the host), runs `warmup`
    untimed iterations, then times `steps` iterations. The seeds are fixed, so every run times the
    same iterations with the same accepted counts."""
    from oracle import jacobi as OJ
    from oracle import oracle as O
    from paper_2512_14681_gb300 import inputs as I

    w = WORKLOADS[DEFAULT_WORKLOAD]
    BLOCK, P_INJECT = w.block, w.p
    shape = I.QWEN7B_BF16
    need = shape.weight_bytes() + (6 << 30)
    avail = os.sysconf("SC_AVPHYS_PAGES") * os.sysconf("SC_PAGE_SIZE")
    if avail < need:
        return None, f"host memory {avail >> 30} GiB < {need >> 30} GiB needed by the 7B oracle"
    prompt = I.prompt_tokens(shape.vocab, w.prompt)[:prompt_len]
    model = O.Model(O.ModelConfig(**shape.oracle_kwargs())).init_random(I.WEIGHT_SEED, I.WEIGHT_STD)
    n_it = steps + warmup
    truth = OJ.generate_ar(model, prompt, n_it * BLOCK + 2 * BLOCK + 2).tokens
    dec = OJ.JacobiDecoder(model, prompt, OJ.GenParams(block_size=BLOCK, init="inject", inject_p=P_INJECT,
                                                       seed=I.INJECT_SEED, max_new=len(truth) - 2 * BLOCK - 2),
                           truth=truth)
    for _ in range(warmup):
        dec.step()
    times, toks = [], 0
    for _ in range(steps):
        t0 = time.perf_counter()
        toks += dec.step().k
        times.append(time.perf_counter() - t0)
    dt = sum(times)
    return dict(value=toks / dt, unit="tokens/s", cores=O.num_threads(), kind="oracle", dtype="f64",
                ms_per_iteration=1000.0 * dt / steps, ms_per_iteration_median=1000.0 * statistics.median(times),
                tokens_per_iteration=toks / steps, iterations=steps,
                sample=f"{steps} timed Jacobi iterations after {warmup} untimed ones (n={BLOCK}, inject p={P_INJECT}, "
                       f"seed {I.INJECT_SEED}) of the 7B-shaped model after a {prompt_len}-token prompt prefill; "
                       f"{toks} tokens in {dt:.1f} s; fp64 arithmetic"), None


def oracle_tiny_run():
    """The oracle's full run of the tiny fp32 decoder (2 layers, d 256, vocabulary 4096; prompt of 32
    tokens, block n = 8 with the repeated last prompt token as initial draft, 64 new tokens)."""
    from oracle import jacobi as OJ
    from oracle import oracle as O
    from paper_2512_14681_gb300 import inputs as I

    shape = I.TINY_F32
    model = O.Model(O.ModelConfig(**shape.oracle_kwargs())).init_random(I.WEIGHT_SEED, I.WEIGHT_STD)
    prompt = I.prompt_tokens(shape.vocab, 32, seed=I.PROMPT_SEED)
    t0 = time.perf_counter()
    res = OJ.generate_jacobi(model, prompt, OJ.GenParams(block_size=8, max_new=64))
    dt = time.perf_counter() - t0
    return dict(value=len(res.tokens) / dt, unit="tokens/s", iterations=len(res.iters),
                ms_per_iteration=1000.0 * dt / max(len(res.iters), 1), dtype="f64",
                sample="tiny fp32 decoder, prompt 32, n=8, 64 new tokens, prefill included")


def run_reference(args, rank):
    if rank != 0:
        return
    # one step = one Jacobi iteration of the oracle on the headline workload's model and parameters
    res, why = oracle_sample(args.steps, args.warmup, args.cpu_baseline_prompt)
    if res is None:
        print(json.dumps({"impl": "reference", "unavailable": why}))
        return
    line = {"impl": "reference", "metric": METRIC, "value": res["value"], "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": res["ms_per_iteration"],
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": DEFAULT_WORKLOAD, "sample": res["sample"]},
            "cpu_baseline": res, "e2e": {"value": res["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0,
                                         "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


# ------------------------------------------------------------------------------------------
# GPU arm
# ------------------------------------------------------------------------------------------
def run_gpu(args, rank, world, local_rank):
    import torch

    from paper_2512_14681_gb300 import inputs as I
    from paper_2512_14681_gb300.jacobi import Context, Gen

    torch.cuda.set_device(local_rank)
    dist = None
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    wl = WORKLOADS[args.workload]
    PROMPT_LEN, BLOCK, NEW, P_INJECT = wl.prompt, wl.block, wl.new, wl.p
    shape = I.SHAPES[wl.shape]
    if args.layers and args.layers != shape.n_layers:
        # reduced-depth copy of the shape: small profiling case only, never a headline number
        shape = dataclasses.replace(shape, n_layers=args.layers, name=f"{shape.name}-{args.layers}layers")
    G = wl.ngram or wl.block
    rows_per_iter = wl.blocks * wl.block + wl.cands * G
    truth_len = NEW + wl.blocks * BLOCK + G + 1
    max_ctx = PROMPT_LEN + truth_len + rows_per_iter + 64
    # prefill in 512-row forwards; decoding needs rows_per_iter rows
    ctx = Context(shape, max_seqs=1, max_ctx=max_ctx, max_rows=max(512, rows_per_iter))
    ctx.init_random_weights(I.WEIGHT_SEED, I.WEIGHT_STD)
    prompt = I.prompt_tokens(shape.vocab, PROMPT_LEN)
    truth = ctx.generate([prompt], Gen(mode="ar", max_new=truth_len)).tokens[0].astype(np.int32)
    gen = Gen(block_size=BLOCK, n_blocks=wl.blocks, spawn_ratio=wl.spawn, pool_size=wl.pool, ngram_len=wl.ngram,
              cand_per_iter=wl.cands, init="inject", inject_p=P_INJECT, seed=I.INJECT_SEED, max_new=NEW)
    d_prompt = torch.from_numpy(prompt).cuda()
    d_truth = torch.from_numpy(truth).cuda().reshape(1, -1)
    d_out = torch.empty((1, NEW), dtype=torch.int32, device="cuda")
    st = ctx.stream

    def step(log_cap=0):
        return ctx.generate_device(d_prompt, [PROMPT_LEN], gen, d_out, d_truth, truth_len, log_cap=log_cap)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    first = step(log_cap=4096)
    assert np.array_equal(d_out.cpu().numpy()[0], truth[:NEW]), "generated tokens differ from the greedy truth"

    def barrier():
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize()

    # ---- timed region: device-resident inputs
    sampler = ClockSampler(local_rank)
    barrier()
    sampler.start()
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    ev0.record(st)
    launches = 0
    iters = 0
    decode_ms = 0.0
    prefill_ms = 0.0
    for _ in range(args.steps):
        o = step()
        launches += o.kernel_launches
        iters += o.iterations
        decode_ms += o.decode_ms
        prefill_ms += o.prefill_ms
    ev1.record(st)
    barrier()
    clocks = sampler.stop()
    total_ms, _, value = aggregate_ranks(ev0.elapsed_time(ev1), NEW * args.steps, dist, "cuda")
    ms_per_step = total_ms / args.steps

    # ---- end to end: host buffers in and out through jf_generate
    barrier()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(st)
    for _ in range(args.steps):
        h = ctx.generate([prompt], gen, truth=truth.reshape(1, -1), log_cap=0)
    e1.record(st)
    barrier()
    assert np.array_equal(h.tokens[0], truth[:NEW])
    _, _, e2e_value = aggregate_ranks(e0.elapsed_time(e1), NEW * args.steps, dist, "cuda")

    # ---- per-kernel timing of the dominant kernel (CUDA events around its launches)
    ctx.set_profiling(True)
    for _ in range(max(1, min(args.steps, 2))):
        step()
    torch.cuda.synchronize()
    gu_ms, gu_n = ctx.kernel_time(0)
    at_ms, at_n = ctx.kernel_time(1)
    class_names = ["gate_up", "attention", "all_gemms", "qkv", "o_proj", "down", "lm_head", None, "rmsnorm", "other"]
    prof = {nm: ctx.kernel_time(i) for i, nm in enumerate(class_names) if nm}
    prof_iters = max(1, prof["lm_head"][1])
    ctx.set_profiling(False)

    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return
    peak, peak_kind = _peaks()
    rows = first.rows.astype(np.float64)
    m_avg = float(rows.mean()) if rows.size else float(BLOCK)
    d, F = shape.d_model, shape.d_ff
    gu_bytes = 2 * F * d * 2 + m_avg * d * 2 + m_avg * F * 2   # weights + activations in + SwiGLU out
    gu_avg_s = gu_ms / max(gu_n, 1) / 1000.0
    achieved = gu_bytes / gu_avg_s / 1e9 if gu_n else None
    # per-iteration roofline: every weight byte + the committed KV read once per iteration
    n_iter = first.iterations
    it_ms = first.decode_ms / max(n_iter, 1)
    # per-iteration device time of each graph replay (CUDA events around it) in the logged step
    it_rep = first.iter_ms if first.iter_ms is not None and len(first.iter_ms) else np.array([it_ms])
    kv_tok = shape.kv_bytes_per_token()
    p_avg = PROMPT_LEN + NEW / 2.0   # committed length averaged over the generation
    it_bytes = shape.weight_bytes() + kv_tok * p_avg
    it_gbs = it_bytes / (it_ms / 1000.0) / 1e9
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic: uniform-random prompt, N(0,0.02) random weights, drafts injected from the model's own "
                "greedy continuation",
        "config": {"workload": args.workload if not args.layers else f"{args.workload} ({args.layers}-layer profiling case)",
                   "layers": shape.n_layers, "prompt": PROMPT_LEN, "block_size": BLOCK, "new_tokens": NEW,
                   "blocks": wl.blocks, "spawn_ratio": wl.spawn, "rr_pool": wl.pool, "ngram": G,
                   "candidates": wl.cands,
                   "rows_per_iteration_max": rows_per_iter,
                   "inject_p": P_INJECT, "kv_page_tokens": 16, "batch": 1,
                   "parallelism": "replicas" if world > 1 else "single-gpu",
                   "l2": "no flush: every step streams 14.1 GB of weights through the 129 MB L2"},
        "e2e": {"value": e2e_value, "unit": "tokens/s", "h2d_bytes_per_step": int(prompt.nbytes + truth.nbytes),
                "d2h_bytes_per_step": int(NEW * 4)},
        "gpu_launches": int(launches),
        "iteration": {"count_per_step": n_iter, "tokens_per_iteration": NEW / max(n_iter, 1), "ms": it_ms,
                      "replay_p50_ms": float(np.median(it_rep)), "replay_p90_ms": float(np.percentile(it_rep, 90)),
                      "prefill_ms": first.prefill_ms, "bytes": it_bytes, "achieved_gbs": it_gbs,
                      "frac_of_" + peak_kind: it_gbs / peak, "frac_of_8tbs": it_gbs / NOMINAL_HBM_GBS},
        "roofline": {"bound": "hbm", "kernel": "gate/up projection GEMM (tcgen05, SwiGLU epilogue)",
                     "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": (achieved / peak) if achieved else None, "traffic": GATEUP_TRAFFIC_BYTES,
                     "bytes_per_launch": gu_bytes, "launches_timed": gu_n, "avg_launch_us": gu_avg_s * 1e6,
                     "peak_kind": peak_kind, "timing": "CUDA events around each launch in a profiled pass of the step"},
        "attention": {"launches_timed": at_n, "avg_launch_us": (at_ms / max(at_n, 1)) * 1000.0},
        "profiled_breakdown_us_per_iteration": {nm: 1000.0 * ms / prof_iters for nm, (ms, n) in prof.items()},
        "clocks": clocks,
    }
    if args.cpu_baseline and world == 1 and args.workload == DEFAULT_WORKLOAD and not args.layers:
        cb, why = oracle_sample(args.cpu_baseline_iters, 1, args.cpu_baseline_prompt)
        if cb is not None:
            cb["tiny_config"] = oracle_tiny_run()
        line["cpu_baseline"] = cb if cb is not None else {"unavailable": why}
    else:
        line["cpu_baseline"] = None
    print(json.dumps(line))
    if dist is not None:
        dist.destroy_process_group()


SWEEP_POINTS = [(P, n, B) for P in (4096, 8192, 16384, 32768) for n in (16, 32, 64, 128) for B in (1, 4)]
# latency versus parallel tokens (the knee of App. D) at P = 4096, one sequence, n = rows
KNEE_ROWS = [16, 32, 64, 128, 192, 256, 320, 384, 512]


def run_sweep(args):
    """Fixed-shape Jacobi iterations on the 7B shape: window mode keeps B*n rows in flight every
    iteration; the latency of an iteration does not depend on the token values."""
    import torch

    from paper_2512_14681_gb300 import inputs as I
    from paper_2512_14681_gb300.jacobi import Context, Gen

    shape = I.QWEN7B_BF16
    peak, peak_kind = _peaks()
    maxP = max(p[0] for p in SWEEP_POINTS)
    ctx = Context(shape, max_seqs=4, max_ctx=maxP + 256, max_rows=512)
    ctx.init_random_weights(I.WEIGHT_SEED, I.WEIGHT_STD)
    pts = []
    points = [(P, n, B, "grid") for P, n, B in SWEEP_POINTS] + [(4096, r, 1, "knee") for r in KNEE_ROWS]
    for P, n, B, kind in points:
        prompts = [I.prompt_tokens(shape.vocab, P, seed=100 + b) for b in range(B)]
        out = ctx.generate(prompts, Gen(block_size=n, mode="window", max_new=args.steps + args.warmup), log_cap=64)
        # median device time of the replays after the warm-up ones (the first iteration of a point also
        # captures and instantiates its graph on the host, which the decode time would include)
        reps = out.iter_ms[args.warmup:] if out.iter_ms is not None and len(out.iter_ms) > args.warmup else None
        it_ms = float(np.median(reps)) if reps is not None else out.decode_ms / max(out.iterations, 1)
        kv = shape.kv_bytes_per_token() * (P + 2) * B
        by = shape.weight_bytes() + kv
        M = n * B
        flops = 2.0 * M * (shape.weight_bytes() / 2) + 4.0 * shape.head_dim * shape.n_heads * P * shape.n_layers * M
        t_bytes = by / (peak * 1e9) * 1e3
        t_flops = flops / 1.936e15 * 1e3
        pts.append({"set": kind, "prompt": P, "block": n, "batch": B, "rows": M, "iteration_ms": it_ms,
                    "iteration_ms_incl_host": out.decode_ms / max(out.iterations, 1), "bytes": by,
                    "gbs": by / (it_ms / 1000.0) / 1e9, "flops": flops,
                    "roofline_ms": max(t_bytes, t_flops), "bound": "hbm" if t_bytes >= t_flops else "tensor",
                    "frac_of_roofline": max(t_bytes, t_flops) / it_ms})
        print(json.dumps(pts[-1]), file=sys.stderr, flush=True)
    med = statistics.median(p["iteration_ms"] for p in pts if p["set"] == "grid")
    print(json.dumps({"metric": "Jacobi-iteration latency sweep on the 7B shape (bf16, window mode)",
                      "value": med, "unit": "ms (median over the grid points)", "n_gpus": 1, "steps": args.steps,
                      "warmup": args.warmup, "higher_is_better": False, "dtype": "bf16", "data": "synthetic",
                      "config": {"workload": "qwen2.5-7b-shape-bf16 sweep P x n x B", "peak_gbs": peak,
                                 "peak_kind": peak_kind, "tensor_peak_tflops": 1936.4},
                      "points": pts}))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", dest="cpu_baseline", action="store_false")
    ap.add_argument("--cpu-baseline-iters", type=int, default=3)
    ap.add_argument("--cpu-baseline-prompt", type=int, default=16,
                    help="prompt tokens the oracle prefills before its timed iterations (1024 = the full prompt, "
                         "several minutes on the host)")
    ap.add_argument("--layers", type=int, default=0, help="decoder layers (0 = the workload's; fewer = profiling case)")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD,
                    help="workload name or alias (" + ", ".join(ALIASES) + "); 'sweep' = fixed-shape latency sweep")
    args = ap.parse_args()
    args.workload = ALIASES.get(args.workload, args.workload)
    if args.workload != "sweep" and args.workload not in WORKLOADS:
        ap.error(f"unknown workload {args.workload}")
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank)
        return
    import __graft_entry__

    __graft_entry__.build()
    if args.workload == "sweep":
        run_sweep(args)
    else:
        run_gpu(args, rank, world, local_rank)


if __name__ == "__main__":
    main()
