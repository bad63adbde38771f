"""Throughput of TADM's anchor-cache sampling loop on GB300.

One step = one whole generation (Alg. 1 over every block) of the workload's
batch, i.e. batch * gen_len generated tokens.  Default workload: "small"
(batch 16, 256 Zipf prompt tokens + 768 masked, 128 reverse steps, K = 4,
d_model 768, 8 anchor + 4 denoiser layers, vocab 32768, bf16).  At N = 1 the
same line also carries "configs": the block-diffusion workload (batch 32,
d_model 2048, 16 + 6 layers, blocks of 32) and the 27 B post-train workload
(batch 8, d_model 5376, 2 + 54 + 6 layers, paired-attention fusion), each
timed over whole generations at K = 1 and its own K, with its GEMMs'
throughput against the tensor and HBM peaks.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload small] [--K 4]
    python bench.py --impl reference ...      # the CPU oracle on a bounded sample

With --gpus N > 1 every rank runs an independent replica on its own GPU
with its own prompts (sequences are independent: no collective on the data
path); value = all ranks' tokens / max-over-ranks time.  Launched without
torchrun, bench.py starts the N local ranks itself.  Prints one JSON line on
rank 0.
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

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "generated tokens/s"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="tadm", choices=["tadm", "reference"])
    ap.add_argument("--workload", default="small")
    ap.add_argument("--K", type=int, default=None, help="anchor refresh interval (default: the workload's)")
    ap.add_argument("--sweep", default="1", help="extra K values timed for the K-sweep (comma list, '' for none)")
    ap.add_argument("--batch", type=int, default=None)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-sample-seconds", type=float, default=20.0)
    ap.add_argument("--T", type=int, default=None,
                    help="override reverse steps per block (short runs for launch-list profiles)")
    ap.add_argument("--G", type=int, default=None, help="override the generation length (short profiling runs)")
    ap.add_argument("--layers", default=None,
                    help="override L_S,L_A,L_D (reduced-depth profiling runs of a wide model, e.g. 0,1,1)")
    ap.add_argument("--no-e2e", action="store_true", help="skip the host-buffer end-to-end leg")
    ap.add_argument("--sampler", default="topk", choices=["topk", "remdm-cap", "remdm-loop", "entropy-bound"],
                    help="with --sweep-workloads: the confidence top-k sampler, ReMDM (App. C.2 settings) or the "
                         "entropy-bound sampler with self-conditioning (App. C.1 settings)")
    ap.add_argument("--fusion-off", action="store_true",
                    help="with --sweep-workloads: run the workloads with the fusion disabled (App. D naive reuse)")
    ap.add_argument("--sweep-workloads", default=None,
                    help="comma list of workloads: print one JSON line per (workload, batch, K) instead")
    ap.add_argument("--sweep-batches", default="", help="batches for the 'sweep' workload (default 1,8,32,128)")
    ap.add_argument("--kernel-bench", default=None,
                    help="time one building block alone instead, e.g. gemm:16384,32768,768")
    ap.add_argument("--qkv-split", type=int, default=None, choices=[0, 1],
                    help="override the model's qkv_split (QKV projection input as bf16 hi + lo)")
    ap.add_argument("--configs", default="block,posttrain",
                    help="at N = 1: workloads also timed whole (K = 1 and the workload's K) and reported under "
                         "'configs' in the same JSON line ('' for none)")
    ap.add_argument("--config-steps", type=int, default=1, help="timed generations per K of each extra workload")
    ap.add_argument("--configs-only", action="store_true",
                    help="time only the extra workloads (one JSON line with their results)")
    ap.add_argument("--config-warmup", type=int, default=2,
                    help="untimed generations per K of each extra workload (the second one captures the CUDA graph)")
    return ap.parse_args()


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def rank_launch_command(gpus: int, argv, port: int):
    """torch.distributed.run command that starts `gpus` local ranks of this
    script with the same arguments (rendezvous on 127.0.0.1)."""
    return [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", f"--nproc-per-node={gpus}",
            "--master-addr", "127.0.0.1", f"--master-port={port}", os.path.abspath(__file__), *argv]


def launch_ranks_if_needed(gpus: int, argv):
    """--gpus N > 1 outside torchrun: start the N ranks here and return their
    exit code.  Inside torchrun, WORLD_SIZE must equal N (None: go on)."""
    env_world = os.environ.get("WORLD_SIZE")
    if env_world is not None:
        if int(env_world) != gpus:
            raise SystemExit(f"bench.py: --gpus {gpus} but WORLD_SIZE={env_world}; launch one rank per GPU")
        return None
    if gpus <= 1:
        return None
    import socket
    with socket.socket() as sk:
        sk.bind(("127.0.0.1", 0))
        port = sk.getsockname()[1]
    return subprocess.call(rank_launch_command(gpus, argv, port))


class Ranks:
    """The replicas of a multi-GPU run: one process per GPU, each generating
    its own sequences, no exchange on the data path.  Only the timing needs
    the group: a barrier on both sides of the timed region and the maximum
    of the per-rank times (tensors on `device`: "cuda" under NCCL, "cpu"
    under gloo)."""

    def __init__(self, world: int, device: str = "cuda"):
        self.world, self.device = world, device

    def barrier(self):
        if self.world > 1:
            import torch.distributed as dist
            dist.barrier()

    def max(self, x: float) -> float:
        if self.world == 1:
            return x
        import torch
        import torch.distributed as dist
        t = torch.tensor([x], dtype=torch.float64, device=self.device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        return float(t.item())


def whole_job_rate(world: int, units_per_step: int, steps: int, ms: float) -> float:
    """Units all ranks processed per second over the slowest rank's time."""
    return world * units_per_step * steps / (ms / 1000.0)


def replica_prompts(w, rank: int):
    """Each replica's own seeded prompts (rank 0 keeps the workload's)."""
    import workloads as wl
    return wl.make_prompts(w, seed=w.seed + 1000 * rank)


# DRAM traffic of the GEMM launches of a small-workload generation, from the
# ncu capture summarised in profiles/small_workload_gemm_traffic.md (mean
# dram__bytes_read.sum + dram__bytes_write.sum per GEMM launch); valid only
# while the GEMM sources are the ones captured (their hash is recorded there).
TRAFFIC_PROFILE = os.path.join(ROOT, "profiles", "small_workload_gemm_traffic.md")
GEMM_SOURCES = ("gemm_tc.cu", "epilogue.cuh", "common.cuh", "splitk.cu")


def gemm_source_hash() -> str:
    import hashlib
    h = hashlib.sha256()
    for f in GEMM_SOURCES:
        with open(os.path.join(ROOT, "paper_2609_37924_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def gemm_traffic():
    """(bytes per GEMM launch, note): the captured figure while the sources
    match, else (None, why)."""
    try:
        text = open(TRAFFIC_PROFILE).read()
    except OSError:
        return None, "no capture"
    vals = {}
    for line in text.splitlines():
        if line.startswith("    ") or ":" not in line:
            continue
        k, _, v = line.partition(":")
        vals[k.strip("`* -")] = v.strip(" `")
    if vals.get("gemm_source_sha16") != gemm_source_hash():
        return None, "GEMM sources changed since the capture"
    try:
        return float(vals["dram_bytes_per_gemm_launch"]), TRAFFIC_PROFILE[len(ROOT) + 1:]
    except (KeyError, ValueError):
        return None, "capture unreadable"


def load_peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        return None


# ----------------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.path = tempfile.mktemp(prefix="clocks", suffix=".csv")
        self.proc = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(gpu_index), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            p = [x.strip() for x in line.split(",")]
            if len(p) < 9:
                continue
            try:
                sm.append(float(p[1]))
                mx = float(p[2])
            except ValueError:
                continue
            for n, v in zip(names, p[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        os.unlink(self.path)
        if not sm:
            return None
        loaded = [x for x in sm if mx and x > 0.5 * mx] or sm
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ----------------------------------------------------------------------------- CPU oracle
def cpu_oracle_sample(workload: str, K: int, budget_s: float, threads: int) -> dict:
    """Time the CPU oracle (as it stands) on one refresh + K denoising steps of
    the workload at batch 1 and extrapolate to a whole generation.  Runs in a
    spawned subprocess so that BLAS threads are set before numpy loads."""
    code = f"""
import json, time, sys
sys.path.insert(0, {ROOT!r})
import numpy as np
import workloads as wl
from oracle import tadm_oracle as O
t_start = time.perf_counter()
w = wl.get_workload({workload!r})
m = w.model
host = wl.make_weights(m, seed=w.seed)
o = O.Oracle(m, host)
prompts = wl.make_prompts(w, batch=1)
T, K = w.steps_per_block, {K}
budget = {budget_s}
t_work = time.perf_counter()
sess = o.new_session(1)
R = w.block_len if w.block_len else w.total_len
if w.block_len:
    t0 = time.perf_counter(); o.prefill(sess, prompts); t_prefill = time.perf_counter() - t0
    z = np.full((1, R), m.vocab - 1, np.int32)
else:
    t_prefill = 0.0
    z = wl.initial_canvas(w, prompts)
t0 = time.perf_counter(); cache = o.anchor_forward(sess, z); t_anchor = time.perf_counter() - t0
steps = []
for n in range(K):
    t0 = time.perf_counter()
    r = o.denoise_step(sess, z, cache, n, T, w.block_len or w.gen_len)
    steps.append(time.perf_counter() - t0)
    z = r["z"]
    if time.perf_counter() - t_work > budget and len(steps) >= 1:
        break
t_step = sum(steps) / len(steps)
# wall covers the whole sample: weights, prompts, prefill, refresh and steps
nb = w.n_blocks
refresh = nb * (-(-T // K))
gen_time = refresh * t_anchor + nb * T * t_step + (t_prefill * (1 + nb) if w.block_len else 0.0)
print(json.dumps(dict(t_anchor=t_anchor, t_step=t_step, steps=len(steps), t_prefill=t_prefill,
                      gen_time=gen_time, tokens=w.gen_len, wall=time.perf_counter() - t_start)))
"""
    env = dict(os.environ, OMP_NUM_THREADS=str(threads), OPENBLAS_NUM_THREADS=str(threads),
               MKL_NUM_THREADS=str(threads), CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env, timeout=1800)
    if r.returncode != 0:
        raise RuntimeError(r.stderr[-2000:])
    return json.loads(r.stdout.strip().splitlines()[-1])


def reference_arm(args):
    """--impl reference: the CPU oracle timed on the host cores."""
    rank, world, _ = dist_env()
    if rank != 0:
        return
    import workloads as wl
    w = wl.get_workload(args.workload)
    K = args.K or w.K
    threads = os.cpu_count() or 1
    times = []
    samp = None
    for i in range(args.warmup + args.steps):
        samp = cpu_oracle_sample(args.workload, K, args.cpu_sample_seconds, threads)
        if i >= args.warmup:
            times.append(samp)
    tok_per_s = [s["tokens"] / s["gen_time"] for s in times]
    value = statistics.median(tok_per_s)
    sample = (f"batch 1 of the '{w.name}' workload: one anchor refresh + {K} denoising steps "
              f"({'with prompt prefill' if w.block_len else 'full canvas'}), extrapolated to the "
              f"{w.steps_per_block * w.n_blocks}-step generation of {w.gen_len} tokens")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "higher_is_better": True,
            # one step = one timed sample (its wall time, weights and set-up included); value divides the
            # generated tokens by the generation time extrapolated from the sample's refresh and step times
            "ms_per_step": 1000.0 * statistics.median([s["wall"] for s in times]),
            "extrapolated_generation_ms": 1000.0 * statistics.median([s["gen_time"] for s in times]),
            "dtype": "f64", "data": "synthetic",
            "config": {"workload": w.name, "batch": 1, "K": K},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": threads, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------- GPU arm
def gpu_arm(args):
    import torch
    import torch.distributed as dist

    import workloads as wl
    from paper_2609_37924_gb300 import TadmModel, upload_weights

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    over = {}
    if args.batch:
        over["batch"] = args.batch
    if args.T:
        over["steps_per_block"] = args.T
    if args.G:
        over["gen_len"] = args.G
    if args.qkv_split is not None:
        over["model_qkv_split"] = bool(args.qkv_split)
    if args.layers:
        ls, la, ld = (int(x) for x in args.layers.split(","))
        over.update(model_n_shared=ls, model_n_anchor=la, model_n_denoise=ld)
    w = wl.get_workload(args.workload, **over)
    K = args.K or w.K
    m = w.model
    B = w.batch
    host_w = wl.make_weights(m, seed=w.seed)
    dev_w = upload_weights(m, host_w)
    del host_w
    prompts = replica_prompts(w, rank)
    bl = w.block_len
    max_rows = max(w.prompt_len, bl) if bl else w.total_len
    tm = TadmModel(m, dev_w, max_batch=B, max_rows=max_rows, max_ctx=w.total_len if bl else 0)
    stream = torch.cuda.current_stream()
    p_dev = torch.from_numpy(prompts).cuda()
    out = torch.empty((B, w.total_len), dtype=torch.int32, device="cuda")

    def one(Kv):
        tm.tadm_generate(p_dev, out, w.gen_len, w.steps_per_block, Kv, bl, stream)

    ranks = Ranks(world, "cuda")

    def barrier():
        ranks.barrier()
        torch.cuda.synchronize()

    def timed(Kv, steps, probe=False, warm=True):
        for _ in range(args.warmup if warm else 0):
            one(Kv)
        tm.tadm_sync_status()
        if probe:
            tm.tadm_probe_enable(400000)
        barrier()
        launches = 0
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ev0.record(stream)
        for _ in range(steps):
            one(Kv)
            launches += tm.tadm_get_counters()["kernel_launches"]
        ev1.record(stream)
        barrier()
        ms = ev0.elapsed_time(ev1)
        brk = tm.tadm_probe_breakdown() if probe else None
        pr = (tm.tadm_probe_read(), brk) if probe else None
        if probe:
            tm.tadm_probe_enable(0)
        tm.tadm_sync_status()
        return ranks.max(ms), launches, pr

    clocks = ClockSampler(local)
    ms, launches, _ = timed(K, args.steps)
    clk = clocks.stop()
    # per-kernel breakdown from a separate generation with every launch
    # bracketed by events (the events add gaps, so the headline is not taken here)
    _, _, probe = timed(K, 1, probe=True, warm=False)
    tokens_per_step = B * w.gen_len
    value = whole_job_rate(world, tokens_per_step, args.steps, ms)
    sweep = {}
    for s in [int(x) for x in args.sweep.split(",") if x.strip()]:
        if s == K:
            continue
        ms_s, _, _ = timed(s, args.steps)
        sweep[str(s)] = whole_job_rate(world, tokens_per_step, args.steps, ms_s)
    sweep[str(K)] = value

    # e2e: public API with host buffers (pinned prompt in, tokens out), copies inside the timed region
    hp = torch.from_numpy(prompts).pin_memory()
    for _ in range(0 if args.no_e2e else args.warmup):
        tm.generate(hp, w.gen_len, w.steps_per_block, K, bl)
    barrier()
    t0 = time.perf_counter()
    res = out
    for _ in range(0 if args.no_e2e else args.steps):
        res = tm.generate(hp, w.gen_len, w.steps_per_block, K, bl)
    barrier()
    e2e_s = ranks.max(max(time.perf_counter() - t0, 1e-9))
    e2e = None if args.no_e2e else {"value": whole_job_rate(world, tokens_per_step, args.steps, 1000.0 * e2e_s),
                                    "unit": "tokens/s", "h2d_bytes_per_step": int(hp.numel() * 4),
                                    "d2h_bytes_per_step": int(res.numel() * 4)}

    peaks = load_peaks()
    (n_launch, gemm_ms, gemm_flops), gemm_kinds = probe
    achieved = gemm_flops / (gemm_ms / 1000.0) / 1e12 if gemm_ms > 0 else None
    if peaks:
        peak, peak_src = peaks["bf16_tflops_sustained"], "measured sustained bf16 (MEASURED_PEAKS.json)"
    else:
        peak, peak_src = 1700.0, "fallback sustained bf16"
    traffic, traffic_src = gemm_traffic()
    alg_bytes = sum(v["bytes"] for k, v in gemm_kinds.items() if k not in ("attention", "norms", "attention_short_rows"))
    roofline = {"bound": "tensor", "kernel": "gemm_tc kernels (tcgen05, all GEMM launches of the step)",
                "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                "frac": (achieved / peak) if achieved else None, "traffic": traffic, "traffic_source": traffic_src,
                "algorithmic_bytes_per_launch": alg_bytes / n_launch if n_launch else None, "peak_source": peak_src,
                "launches_timed": n_launch, "gemm_ms_per_step": gemm_ms,
                "gemm_share_of_step": gemm_ms / (ms / args.steps) if ms else None,
                "probe": "one extra generation with events around every GEMM / attention / norm launch",
                "by_epilogue": {k: {"ms_per_step": v["ms"], "tflops": round(v["tflops"], 1),
                                    "launches_per_step": v["launches"]}
                                for k, v in gemm_kinds.items() if k not in ("attention", "norms", "attention_short_rows")},
                # the other probed launches of the step: attention (FLOP/s) and the norms
                "others": {k: {"ms_per_step": v["ms"], "share_of_step": v["ms"] / (ms / args.steps) if ms else None,
                               "tflops": round(v["tflops"], 1) if k.startswith("attention") else None,
                               "launches_per_step": v["launches"]}
                           for k, v in gemm_kinds.items() if k in ("attention", "norms", "attention_short_rows")}}

    line = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if m.dtype == "bf16" else "f32",
            "data": "synthetic (seeded random-init weights N(0,0.02), Zipf-1.1 prompt ids)",
            "config": {"workload": w.name, "batch": B, "prompt_len": w.prompt_len, "gen_len": w.gen_len,
                       "steps_per_block": w.steps_per_block, "block_len": bl, "K": K, "d_model": m.d_model,
                       "layers_anchor": m.n_anchor, "layers_denoise": m.n_denoise, "vocab": m.vocab,
                       "qkv_split": bool(m.qkv_split),
                       "parallelism": f"replicas x{world}",
                       "l2": "inputs larger than L2 (weights + activations per step >> 129 MB)"},
            "k_sweep_tokens_per_s": sweep, "roofline": roofline, "clocks": clk,
            "e2e": e2e, "gpu_launches": launches}
    # the other configurations, timed whole by this same run (N = 1 only)
    del tm, dev_w
    torch.cuda.empty_cache()
    if world == 1 and args.configs:
        line["configs"] = {}
        for name in [x for x in args.configs.split(",") if x]:
            try:
                line["configs"][name] = config_leg(name, args.config_steps, args.config_warmup, peaks, local)
            except Exception as e:  # context for the headline; the line still prints
                line["configs"][name] = {"error": str(e)[-300:]}
            torch.cuda.empty_cache()
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        try:
            threads = os.cpu_count() or 1
            s = cpu_oracle_sample(args.workload, K, args.cpu_sample_seconds, threads)
            s1 = cpu_oracle_sample(args.workload, K, args.cpu_sample_seconds, 1)
            line["cpu_baseline"] = {
                "value": s["tokens"] / s["gen_time"], "unit": "tokens/s", "cores": threads, "kind": "oracle",
                "sample": (f"batch 1: one anchor refresh ({s['t_anchor']:.2f} s) + {s['steps']} denoising steps "
                           f"({s['t_step']:.2f} s each) of the '{w.name}' workload, extrapolated to the "
                           f"{w.steps_per_block * w.n_blocks}-step generation of {w.gen_len} tokens"),
                "single_thread": {"value": s1["tokens"] / s1["gen_time"], "unit": "tokens/s", "cores": 1,
                                  "sample": f"the same sample on one thread (refresh {s1['t_anchor']:.2f} s, "
                                            f"{s1['steps']} steps of {s1['t_step']:.2f} s)"}}
        except Exception as e:  # the baseline is context; the GPU line still prints
            line["cpu_baseline"] = {"error": str(e)[-300:]}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def config_leg(name: str, steps: int, warmup: int, peaks, local: int) -> dict:
    """Whole generations of another workload at K = 1 and its own K: tokens/s,
    the speedup over K = 1 and, from one probed generation at its K, the GEMMs'
    throughput against the tensor peak and their algorithmic bytes against
    HBM bandwidth (the weight-streaming configurations are bound by the
    latter).  Each timed generation includes the prompt prefill and every
    block's commit pass."""
    import torch

    import workloads as wl
    from paper_2609_37924_gb300 import TadmModel, upload_weights

    w = wl.get_workload(name)
    m, B, bl = w.model, w.batch, w.block_len
    t0 = time.perf_counter()
    dev_w = upload_weights(m, wl.make_weights(m, seed=w.seed))
    t_weights = time.perf_counter() - t0
    tm = TadmModel(m, dev_w, max_batch=B, max_rows=max(w.prompt_len, bl) if bl else w.total_len,
                   max_ctx=w.total_len if bl else 0)
    p = torch.from_numpy(wl.make_prompts(w)).cuda()
    out = torch.empty((B, w.total_len), dtype=torch.int32, device="cuda")
    stream = torch.cuda.current_stream()
    res, ms_gen = {}, {}
    clocks = ClockSampler(local)
    for Kv in sorted({1, w.K}):
        for _ in range(warmup):
            tm.tadm_generate(p, out, w.gen_len, w.steps_per_block, Kv, bl, stream)
        tm.tadm_sync_status()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(steps):
            tm.tadm_generate(p, out, w.gen_len, w.steps_per_block, Kv, bl, stream)
        e1.record(stream)
        torch.cuda.synchronize()
        ms_gen[Kv] = e0.elapsed_time(e1) / steps
        res[Kv] = B * w.gen_len / (ms_gen[Kv] / 1000.0)
    clk = clocks.stop()
    tm.tadm_sync_status()
    valid = bool((out != m.mask_id).all())
    # one probed generation at the workload's K (events around every launch)
    tm.tadm_probe_enable(1000000)
    tm.tadm_generate(p, out, w.gen_len, w.steps_per_block, w.K, bl, stream)
    kinds = tm.tadm_probe_breakdown()
    tm.tadm_probe_enable(0)
    tm.tadm_sync_status()
    gemm = [v for k, v in kinds.items() if k not in ("attention", "norms", "attention_short_rows")]
    g_ms = sum(v["ms"] for v in gemm)
    g_fl = sum(v["flops"] for v in gemm)
    g_by = sum(v["bytes"] for v in gemm)
    tf_peak = peaks["bf16_tflops_sustained"] if peaks else 1700.0
    bw_peak = peaks["hbm_gbs"] if peaks else 6800.0
    tflops = g_fl / (g_ms / 1000.0) / 1e12 if g_ms > 0 else None
    gbs = g_by / (g_ms / 1000.0) / 1e9 if g_ms > 0 else None
    bound = "hbm" if (gbs or 0) / bw_peak > (tflops or 0) / tf_peak else "tensor"
    leg = {"workload": name, "batch": B, "prompt_len": w.prompt_len, "gen_len": w.gen_len, "block_len": bl,
           "steps_per_block": w.steps_per_block, "d_model": m.d_model,
           "layers": [m.n_shared, m.n_anchor, m.n_denoise], "vocab": m.vocab,
           "tokens_per_s": {str(k): v for k, v in res.items()},
           "ms_per_generation": {str(k): v for k, v in ms_gen.items()},
           "vs_K1": res[w.K] / res[1], "timed_generations": steps, "warmup": warmup,
           "all_unmasked": valid, "weights_s": round(t_weights, 1), "clocks": clk,
           "roofline": {"bound": bound, "kernel": "gemm_tc kernels (all GEMM launches of one generation at K="
                                                  f"{w.K})",
                        "tflops": tflops, "tensor_peak": tf_peak, "tensor_frac": tflops / tf_peak if tflops else None,
                        "gbs": gbs, "hbm_peak": bw_peak, "hbm_frac": gbs / bw_peak if gbs else None,
                        "gemm_ms_per_generation": g_ms,
                        "gemm_share": g_ms / ms_gen[w.K] if ms_gen.get(w.K) else None,
                        "launches": int(sum(v["launches"] for v in gemm)),
                        "peak_source": "MEASURED_PEAKS.json (sustained bf16, HBM copy)" if peaks else "fallback"},
           "others_ms_per_generation": {k: v["ms"] for k, v in kinds.items()
                                        if k in ("attention", "norms", "attention_short_rows")},
           "gemm_by_epilogue": {k: {"ms": round(v["ms"], 2), "launches": v["launches"],
                                    "tflops": round(v["tflops"], 1),
                                    "gbs": round(v["bytes"] / (v["ms"] / 1e3) / 1e9, 1) if v["ms"] > 0 else None}
                                for k, v in kinds.items() if k not in ("attention", "norms", "attention_short_rows")}}
    tm.close()
    del tm, dev_w
    return leg


def kernel_bench(args):
    """Times one building block alone through the C ABI (for isolated ncu
    captures of the GEMM): C[M, N] = A[M, K] B[N, K]^T, bf16 in, bf16 out."""
    import torch
    from paper_2609_37924_gb300 import tadm
    kind, shape = args.kernel_bench.split(":")
    g = torch.Generator(device="cuda").manual_seed(0)
    if kind == "attnctx":
        # attnctx:B,H,Hkv,R,ctx,hd  R canvas rows over ctx committed keys + themselves (block-step shape), bf16
        B, H, Hkv, R, ctx, hd = (int(x) for x in shape.split(","))
        stride = (ctx + R + 7) // 8 * 8
        q = torch.randn((B, H, R, hd), device="cuda", generator=g).to(torch.bfloat16)
        k = torch.randn((B, Hkv, stride, hd), device="cuda", generator=g).to(torch.bfloat16)
        v = torch.randn((B, Hkv, hd, stride), device="cuda", generator=g).to(torch.bfloat16)
        o = torch.empty((B * R, H * hd), device="cuda", dtype=torch.bfloat16)
        run = lambda: tadm.tadm_attention(q, k, v, o, H, Hkv, R, ctx, False, dtype=1)  # noqa: E731
        flops = 4.0 * B * H * R * (ctx + R) * hd
    elif kind == "attn":
        # attn:B,H,Hkv,R,hd  bidirectional attention of R rows (no context), bf16
        B, H, Hkv, R, hd = (int(x) for x in shape.split(","))
        q = torch.randn((B, H, R, hd), device="cuda", generator=g).to(torch.bfloat16)
        k = torch.randn((B, Hkv, R, hd), device="cuda", generator=g).to(torch.bfloat16)
        v = torch.randn((B, Hkv, R, hd), device="cuda", generator=g).to(torch.bfloat16)
        o = torch.empty((B * R, H * hd), device="cuda", dtype=torch.bfloat16)
        run = lambda: tadm.tadm_attention(q, k, v, o, H, Hkv, R, 0, False, dtype=1)  # noqa: E731
        flops = 4.0 * B * H * R * R * hd
    elif kind == "ebrow":
        # ebrow:rows,V  one entropy-bound sampler step (Alg. 2) on fp32 logits of `rows` positions of one
        # sequence: per-position softmax/entropy/draw with p written as bf16, then the accept kernel
        rows, V = (int(x) for x in shape.split(","))
        logits = torch.randn((rows, V), device="cuda", generator=g) * 3.0
        z = torch.zeros((1, rows), dtype=torch.int32, device="cuda")
        ent = torch.empty(rows, dtype=torch.float32, device="cuda")
        probs = torch.empty((rows, V), dtype=torch.bfloat16, device="cuda")
        run = lambda: tadm.tadm_eb_update(z, logits, 0, V - 1, 0.6, 0.1, False, 1, 0, ent, probs)  # noqa: E731
        flops = 0.0
    else:
        M, N, K = (int(x) for x in shape.split(","))
        A = torch.randn((M, K), device="cuda", generator=g).to(torch.bfloat16)
        Bm = torch.randn((N, K), device="cuda", generator=g).to(torch.bfloat16)
        C = torch.empty((M, N), device="cuda", dtype=torch.bfloat16)
        run = lambda: tadm.tadm_gemm(A, Bm, C, dtype=1)  # noqa: E731
        flops = 2.0 * M * N * K
    for _ in range(args.warmup):
        run()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(args.steps):
        run()
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / args.steps
    line = {"kernel": kind, "shape": shape, "ms": ms, "tflops": flops / (ms / 1000.0) / 1e12}
    if kind == "attnctx":   # K and V bytes read once per launch
        line["kv_gbs"] = 2 * k.numel() * (ctx + R) / stride * 2 / (ms / 1000.0) / 1e9
    if kind == "ebrow":     # algorithmic bytes: the fp32 logits read once, p written once as bf16
        line["gbs"] = rows * V * (4 + 2) / (ms / 1000.0) / 1e9
        del line["tflops"]
    print(json.dumps(line), flush=True)


def workload_sweep(args):
    """Generated tokens/s of each workload for every K of its sweep (one line each)."""
    import torch

    import workloads as wl
    from paper_2609_37924_gb300 import TadmModel, upload_weights

    torch.cuda.set_device(0)
    peaks = load_peaks()
    peak = peaks["bf16_tflops_sustained"] if peaks else 1700.0
    for name in args.sweep_workloads.split(","):
        # --fusion-off: the same workload with the fusion disabled (the naive
        # stale-anchor reuse baseline of App. D), for the fusion-cost ablation
        base = wl.get_workload(name, **({"model_fusion": "none"} if args.fusion_off else {}))
        batches = [base.batch]
        if name == "sweep":
            batches = [int(b) for b in (args.sweep_batches or "1,8,32,128").split(",")]
        m = base.model
        t0 = time.perf_counter()
        dev_w = upload_weights(m, wl.make_weights(m, seed=base.seed))
        t_w = time.perf_counter() - t0
        for B in batches:
            w = wl.get_workload(name, batch=B, **({"model_fusion": "none"} if args.fusion_off else {}))
            bl = w.block_len
            tm = TadmModel(m, dev_w, max_batch=B, max_rows=max(w.prompt_len, bl) if bl else w.total_len,
                           max_ctx=w.total_len if bl else 0)
            p = torch.from_numpy(wl.make_prompts(w)).cuda()
            out = torch.empty((B, w.total_len), dtype=torch.int32, device="cuda")
            res = {}
            remdm = args.sampler.startswith("remdm")
            if remdm:   # ReMDM sampler (App. C.2 settings): logits of the masked rows per step
                if bl:
                    raise SystemExit("the ReMDM sampler runs single-block workloads")
                scratch = torch.empty((B * w.gen_len, m.vocab), dtype=torch.float32, device="cuda")
                kind = args.sampler.split("-")[1]
                eta = 0.04 if kind == "cap" else 0.02
            ebs = args.sampler == "entropy-bound"
            if ebs:     # App. C.1: eta 0.1, tau 0.8 -> 0.4, self-conditioning on
                if bl:
                    raise SystemExit("the entropy-bound sampler runs single-block workloads")
                scratch = torch.empty(tm.tadm_eb_scratch_bytes(B, w.gen_len, True), dtype=torch.uint8,
                                      device="cuda")

            def gen(K):
                if ebs:
                    tm.tadm_generate_entropy_bound(p, out, w.gen_len, w.steps_per_block, K, 0.1, 0.8, 0.4, 1234,
                                                   scratch, True)
                elif remdm:
                    tm.tadm_generate_remdm(p, out, w.gen_len, w.steps_per_block, K, kind, eta, 0.9, 1234, scratch)
                else:
                    tm.tadm_generate(p, out, w.gen_len, w.steps_per_block, K, bl)
            for K in (w.k_sweep or (w.K,)):
                # the second identical top-k call captures the CUDA graph; the other samplers run eagerly
                for _ in range(max(2 if args.sampler == "topk" else 1, args.warmup)):
                    gen(K)
                tm.tadm_sync_status()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                torch.cuda.synchronize()
                e0.record()
                for _ in range(args.steps):
                    gen(K)
                e1.record()
                tm.tadm_sync_status()
                ms = e0.elapsed_time(e1) / args.steps
                c = tm.tadm_get_counters()
                res[K] = B * w.gen_len / (ms / 1000.0)
                # one more generation with every GEMM launch bracketed by events (up to 400000 launches)
                tm.tadm_probe_enable(400000)
                gen(K)
                n_l, g_ms, g_fl = tm.tadm_probe_read()
                tm.tadm_probe_enable(0)
                tm.tadm_sync_status()
                g_tf = g_fl / (g_ms / 1000.0) / 1e12 if g_ms > 0 else None
                done = out.cpu().numpy()
                valid = bool((done != m.mask_id).all())
                print(json.dumps({"workload": name, "fusion": m.fusion, "sampler": args.sampler, "all_unmasked": valid,
                                  "batch": B, "K": K, "tokens_per_s": res[K],
                                  "ms_per_generation": ms,
                                  "vs_K1": res[K] / res[1] if 1 in res else None, "anchor_calls": c["anchor_calls"],
                                  "denoise_steps": c["denoise_steps"], "commit_passes": c["commit_passes"],
                                  "gpu_launches": c["kernel_launches"], "weights_s": round(t_w, 1),
                                  "gemm": {"tflops": g_tf, "frac_of_sustained": (g_tf / peak) if g_tf else None,
                                           "launches_probed": n_l, "ms_probed": g_ms}}), flush=True)
            tm.close()
            del tm
            torch.cuda.empty_cache()
        del dev_w
        torch.cuda.empty_cache()


def main():
    args = parse()
    rc = launch_ranks_if_needed(args.gpus, sys.argv[1:])
    if rc is not None:
        sys.exit(rc)
    if args.sweep_workloads:
        import __graft_entry__
        __graft_entry__.build()
        workload_sweep(args)
        return
    if args.kernel_bench:
        import __graft_entry__
        __graft_entry__.build()
        kernel_bench(args)
        return
    if args.configs_only:
        import __graft_entry__
        import torch
        __graft_entry__.build()
        torch.cuda.set_device(0)
        print(json.dumps({name: config_leg(name, args.config_steps, args.config_warmup, load_peaks(), 0)
                          for name in args.configs.split(",") if name}), flush=True)
        return
    if args.impl == "reference":
        reference_arm(args)
    else:
        import __graft_entry__
        __graft_entry__.build()
        gpu_arm(args)


if __name__ == "__main__":
    main()
