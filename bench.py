"""Benchmark of the PS-PPO LM-head update pass on GB300.

One step = one pass of the whole hot path over one synthetic rollout batch of the
7B-shaped workload (16 prompts x 8 completions, lognormal lengths around 2048 clipped
to [128, 8192], d = 3584, V = 152064, bf16): cutoff sampling -> prefix packing ->
fused LM-head forward -> fused LM-head backward (dH and dW). Every step draws new
cutoffs (the Philox step counter advances), so N varies from step to step.

value: prefix tokens/s, whole job (sum of packed rows over all steps and ranks divided
by the max over ranks of the device-timed region). The credited work of a step is
6 N d V FLOPs (forward GEMM, dH, dW). By default the forward keeps its logits in the
logit store where the device memory holds it (about 60 GB at the 7B workload), and the
backward turns them into dZ in place instead of recomputing them (executing 6 N d V
rather than 8 N d V); --logits recompute times the recomputing backward, and the line's
recompute_control does so on the same batch in every run.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference|torch]

With --gpus N > 1 (launched by torchrun) the step is data-parallel (weak scaling): every rank
holds its own batch of the workload's P prompts (global batch N x P), draws the cutoffs of its
completions by their global index (traj_base = rank x P x K) with the global loss scale
1/(N P K), and after the backward dW and the loss are summed over the ranks (NCCL all-reduce,
inside the timed step). --replicas runs N independent replicas without the exchange. --impl reference times the CPU float64 oracle on bounded samples of
the same workload, on the host cores. --impl torch (context only) runs the head of the same step
in eager PyTorch with materialised logits.
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

WORKLOAD = "7b"
MEASURED_PEAKS = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}

# DRAM bytes (read + write) per launch of the forward GEMM on the 7b workload, the mean of the
# launches in profiles/lmhead_pass_7b_launch_list.md: the forward keeping its logits 72.04 GB read +
# 64.18 GB written (its algorithmic write is the logit store, 64.5 GB); the plain forward None until
# its current kernel is captured at that size. Reset an entry whenever that kernel or its schedule
# changes.
FWD_GEMM_TRAFFIC = {("7b", "FwdLseEpi"): None, ("7b", "FwdLseStoreEpi"): 136.22e9}


def describe(cfg) -> str:
    law = (f"lognormal(median {cfg.len_median}) clipped [{cfg.len_lo}, {cfg.len_hi}]" if cfg.len_law == "lognormal"
           else f"uniform [{cfg.len_lo}, {cfg.len_hi}]")
    return (f"{cfg.name}: {cfg.P} prompts x {cfg.K} completions, lengths {law}, d={cfg.d}, V={cfg.V}, "
            f"{cfg.dtype}, Beta cutoff pmf, eps={cfg.eps}, mode={cfg.mode}")


def _peaks():
    try:
        with open(MEASURED_PEAKS) as f:
            p = json.load(f)
        return p, "measured"
    except Exception:
        return FALLBACK_PEAKS, "fallback"


SLOWDOWNS = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown")


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons while the timed region runs."""
    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        rows = []
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) != 7:
                continue
            try:
                rows.append((float(parts[0]), float(parts[1]), float(parts[2]), parts[3:]))
            except ValueError:
                continue
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, _, fl in rows for i, v in enumerate(fl) if v.lower() == "active"})
        loaded = [r for r in rows if r[2] > 200.0] or rows
        return {"sm_mhz": float(np.median([r[0] for r in loaded])), "sm_max_mhz": rows[0][1],
                "reasons": reasons, "samples": len(rows), "power_w_max": max(r[2] for r in rows)}


def _dist():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def logit_store_rows(args, cfg, b, dev):
    """Rows of the logit store: 0 (recompute the logits in the backward), or as many of the batch's
    sum of lengths (the largest N a step can have) as fit in the device memory left after the pass's
    other buffers, with a margin."""
    import torch

    from paper_2606_29758_gb300 import ps_lmhead_logit_store_size
    if args.logits == "recompute" or cfg.dtype != "bf16":
        return 0
    free, _ = torch.cuda.mem_get_info(dev)
    rows, d, V = b.total_len, cfg.d, cfg.V
    other = (rows * d * 6.0                          # packed hidden rows (bf16) and dH (f32)
             + rows * ((V + 255) // 256 * 8.0 + 64)  # forward partials, per-row vectors
             + min(args.chunk_rows, rows) * V * 2.0  # the recompute path's dZ chunk
             + V * d * 4.0                           # dW
             + rows * (d * 4.0 + 32)                 # the end-to-end stager's two input buffers
             + rows * 3e3                            # the design stage's proxy and top-16 buffers
             + 20e9)                                 # margin
    per_row = ps_lmhead_logit_store_size(1 << 16, V) / (1 << 16)
    return int(max(0, min(rows, (free - other) // per_row)))


def run_ours(args):
    import torch
    import torch.distributed as dist

    from paper_2606_29758_gb300 import DataParallelUpdate, InputStager, PassShape, UpdatePass
    from synthetic import get_config, make_batch

    world, rank, local = _dist()
    torch.cuda.set_device(local)
    dev = f"cuda:{local}"
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device(dev))
    cfg = get_config(args.config)
    b = make_batch(cfg, device=dev)
    D = b.dev
    tdtype = torch.bfloat16 if cfg.dtype == "bf16" else torch.float32
    store_rows = logit_store_rows(args, cfg, b, dev)
    shape = PassShape(cfg.P, cfg.K, b.T_max, cfg.d, cfg.V, b.total_len, tdtype, args.chunk_rows, store_rows)
    # data-parallel: every rank's completions are a slice of one global batch of world x P prompts
    dp = world > 1 and not args.replicas
    up = UpdatePass(shape, device=dev, eps=cfg.eps, loss_scale=cfg.loss_scale / world if dp else cfg.loss_scale)
    dpu = DataParallelUpdate(up, traj_base=rank * cfg.B if dp else 0)
    stream = torch.cuda.current_stream()
    seed = cfg.seed

    def step(i, ev=None):
        if ev is not None:
            ev[0].record(stream)
        up.sample(D["q"], D["L"], seed, i, traj_base=dpu.traj_base)
        if ev is not None:
            ev[1].record(stream)
        n = up.pack(D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"])
        if ev is not None:
            ev[2].record(stream)
        up.forward(D["W"])
        if ev is not None:
            ev[3].record(stream)
        up.backward(D["W"])
        if ev is not None:
            ev[4].record(stream)
        if dp:
            dpu.exchange()
        if ev is not None:
            ev[5].record(stream)
        return n

    def barrier():
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    for i in range(args.warmup):
        step(1000 + i)
    up.check_status()
    barrier()

    def timed_region(base):
        clocks = ClockSampler(local)
        clocks.start()
        time.sleep(0.3)
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(6)] for _ in range(args.steps)]
        barrier()
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        step_rows = []
        for i in range(args.steps):
            step_rows.append(step(base + i, evs[i]))
        t1.record(stream)
        barrier()
        clk = clocks.stop()
        up.check_status()
        per = np.array([[e[j].elapsed_time(e[j + 1]) for j in range(5)] for e in evs])   # sample, pack, fwd, bwd, exchange
        return t0.elapsed_time(t1), step_rows, per, clk

    ms, step_rows, per, clk = timed_region(0)
    # A timed region that saw a thermal or hardware slowdown is not a valid number: measure once more
    # (every rank takes the same decision).
    bad = float(any(r in SLOWDOWNS for r in clk.get("reasons", [])))
    if world > 1:
        t = torch.tensor([bad], device=dev, dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        bad = float(t.item())
    if bad > 0:
        first = clk
        ms, step_rows, per, clk = timed_region(500)
        clk["remeasured_after"] = first.get("reasons", [])
    rows = sum(step_rows)
    # the last timed step's rows: how many the clip switched off (coef = 0 with A != 0), and the
    # packing rate (hidden rows read and written; the pack call includes its host sync)
    n_last = step_rows[-1]
    coef_last, adv_last = up.coef[:n_last], up.adv[:n_last]
    clipped = int(((coef_last == 0) & (adv_last != 0)).sum().item())
    pass_stats = {"rows_last_step": n_last, "clip_fraction": clipped / max(n_last, 1),
                  "zero_advantage_fraction": float((adv_last == 0).float().mean().item()),
                  "pack_gbs": 2.0 * float(np.mean(step_rows)) * cfg.d * (2 if cfg.dtype == "bf16" else 4)
                  / (float(per[:, 1].mean()) * 1e-3) / 1e9,
                  "sample_us": float(per[:, 0].mean()) * 1e3,
                  # algorithmic bytes of one sampler call: the masses q (8 B) read and the weight table
                  # (4 B) written per (prompt, step), lengths read and (H, n) written per completion
                  "sample_gbs": (12.0 * cfg.P * b.T_max + 12.0 * cfg.B) / (float(per[:, 0].mean()) * 1e-3) / 1e9,
                  "sample_bytes": 12 * cfg.P * b.T_max + 12 * cfg.B,
                  "peak_device_memory_gb": torch.cuda.max_memory_allocated() / 1e9}

    ms_max = ms
    rows_all = rows
    if world > 1:
        t = torch.tensor([ms], device=dev, dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms_max = float(t.item())
        r = torch.tensor([rows], device=dev, dtype=torch.float64)
        dist.all_reduce(r)
        rows_all = int(r.item())

    # ---- end-to-end: host (pinned) inputs -> device -> pass -> loss back to the host, every step.
    # The library's InputStager copies batch i + 1 on a copy stream while the pass runs on batch i;
    # every step's copy and loss read stay inside the timed region.
    host = {k: D[k].cpu().pin_memory() for k in ("q", "L", "R", "tok_full", "oldlogp_full", "hid_full")}
    stager = InputStager(host, device=dev)
    loss_h = torch.empty(args.steps + 1, dtype=torch.float64).pin_memory()
    h2d = stager.nbytes

    def e2e_run(n_steps, base):
        total = 0
        j = stager.stage(host)
        for i in range(n_steps):
            X = stager.acquire(j, stream)
            nxt = stager.stage(host) if i + 1 < n_steps else None
            up.sample(X["q"], X["L"], seed, base + i, traj_base=dpu.traj_base)
            total += up.pack(X["L"], X["R"], X["tok_full"], X["oldlogp_full"], X["hid_full"])
            up.forward(D["W"])
            up.backward(D["W"])
            if dp:
                dpu.exchange()
            stager.release(j, stream)
            loss_h[i].copy_(up.loss[0], non_blocking=True)
            stream.synchronize()
            j = nxt
        return total

    e2e_run(1, 2000)
    barrier()
    e0 = time.perf_counter()
    e_rows = e2e_run(args.steps, 0)
    barrier()
    e_ms = (time.perf_counter() - e0) * 1e3
    if world > 1:
        t = torch.tensor([e_ms], device=dev, dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        e_ms = float(t.item())
        r = torch.tensor([e_rows], device=dev, dtype=torch.float64)
        dist.all_reduce(r)
        e_rows = int(r.item())
    # the copy alone, for the record: one batch host -> device with nothing else running
    c0 = torch.cuda.Event(enable_timing=True)
    c1 = torch.cuda.Event(enable_timing=True)
    c0.record(stream)
    for k in host:
        stager.bufs[0][k].copy_(host[k], non_blocking=True)
    c1.record(stream)
    torch.cuda.synchronize()
    h2d_ms = c0.elapsed_time(c1)

    # ---- control: the same batch with every completion kept whole (H = L, all weights 1), the
    # untruncated update that prefix sampling replaces; timed apart from the headline.
    def full_control_run():
        from paper_2606_29758_gb300 import PS_MODE_FULL
        mode0 = up.mode
        up.mode = PS_MODE_FULL
        try:
            for i in range(2):
                step(3000 + i)
            barrier()
            f0 = torch.cuda.Event(enable_timing=True)
            f1 = torch.cuda.Event(enable_timing=True)
            f_steps = 3
            f0.record(stream)
            f_rows = sum(step(3100 + i) for i in range(f_steps))
            f1.record(stream)
            barrier()
        finally:
            up.mode = mode0
        up.check_status()
        f_ms = f0.elapsed_time(f1) / f_steps
        return {"ms_per_step": f_ms, "rows_per_step": f_rows / f_steps,
                "tokens_per_s": f_rows / (f_ms * f_steps * 1e-3),
                "step_time_ratio_full_over_prefix": f_ms / (ms / args.steps),
                "note": "same batch, every completion kept whole (H = L, weights 1); 3 timed steps"}

    # the parts after the headline are context: on one GPU a failure in one is recorded, not fatal
    # (with several ranks it stays fatal, so that no rank is left waiting at a barrier)
    def optional(fn, *a):
        if world > 1:
            return fn(*a)
        try:
            return fn(*a)
        except Exception as e:          # noqa: BLE001
            return {"error": f"{type(e).__name__}: {e}"}

    full_control = optional(full_control_run)

    # ---- control: the same steps with the logits recomputed in the backward instead of kept
    def recompute_control_run():
        up.use_store = False
        try:
            for i in range(2):
                step(3500 + i)
            barrier()
            r0 = torch.cuda.Event(enable_timing=True)
            r1 = torch.cuda.Event(enable_timing=True)
            r_steps = 3
            r0.record(stream)
            r_rows = sum(step(3600 + i) for i in range(r_steps))
            r1.record(stream)
            barrier()
        finally:
            up.use_store = True
        up.check_status()
        r_ms = r0.elapsed_time(r1) / r_steps
        return {"ms_per_step": r_ms, "tokens_per_s": r_rows / (r_ms * r_steps * 1e-3),
                "step_time_ratio_over_store": r_ms / (ms / args.steps),
                "note": "the same prefix steps with the logits recomputed by the backward (chunks of "
                        f"{args.chunk_rows} rows) instead of kept in the logit store; 3 timed steps"}

    recompute_control = optional(recompute_control_run) if store_rows > 0 else None

    # ---- context: the same step with the head split into vocabulary shards (VocabParallelHead), the
    # shards run one after another on this device: what the split itself costs
    def vocab_parallel_run(S):
        from paper_2606_29758_gb300 import VocabParallelHead, vocab_shards
        shards = vocab_shards(cfg.V, S)
        # the shards keep their logits when the whole-head step does (stores of their own, beside the
        # whole head's)
        vp = VocabParallelHead(shards, b.total_len, cfg.d, cfg.V, tdtype, device=dev, eps=cfg.eps,
                               loss_scale=up.loss_scale, bwd_chunk_rows=args.chunk_rows, store=store_rows > 0)
        W = D["W"]

        def vstep(i):
            up.sample(D["q"], D["L"], seed, i, traj_base=dpu.traj_base)
            n = up.pack(D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"])
            for r, (v0, Vs) in enumerate(shards):
                vp.stats(r, n, up.hid, W[v0:v0 + Vs], up.tok)
            vp.forward(n, up.tok, up.oldlogp, up.adv, up.w)
            for r, (v0, Vs) in enumerate(shards):
                vp.backward(r, n, up.hid, W[v0:v0 + Vs], up.tok, up.dH, up.dW[v0:v0 + Vs], add_to_dH=r > 0)
            return n

        for i in range(2):
            vstep(4000 + i)
        barrier()
        v0e, v1e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        v0e.record(stream)
        v_rows = sum(vstep(i) for i in range(3))
        v1e.record(stream)
        barrier()
        v_ms = v0e.elapsed_time(v1e) / 3
        del vp
        return {"shards": S, "ms_per_step": v_ms, "tokens_per_s": v_rows / (v_ms * 3e-3),
                "step_time_ratio_over_whole_head": v_ms / (ms / args.steps),
                "logits": "kept in a store per shard" if store_rows > 0 else "recomputed",
                "note": "the same steps with W split into vocabulary shards run one after another on this device "
                        "(logit statistics per shard, the forward from them, each shard's backward); 3 timed steps"}

    vocab_parallel = optional(vocab_parallel_run, args.vocab_shards) if args.vocab_shards > 0 else None
    if args.no_design:
        design = None
    elif cfg.dtype != "bf16":
        design = {"skipped": "the score proxy of the design stage takes bf16 inputs only"}
    else:
        design = optional(time_design_stage, cfg, b, dev, stream)

    peaks, src = _peaks()
    d, V = cfg.d, cfg.V
    mean_rows = rows / args.steps
    stored = [n <= store_rows for n in step_rows]      # steps whose forward kept the logits
    all_stored = all(stored)
    executed = 6.0 if all_stored else 8.0               # executed FLOPs per row, in units of d V
    t_fwd = float(per[:, 2].mean()) * 1e-3
    fwd_flops = 2.0 * mean_rows * d * V
    peak_tf = peaks["bf16_tflops_sustained"]
    achieved_tf = fwd_flops / t_fwd / 1e12
    step_s = ms / args.steps * 1e-3
    credited_tf = 6.0 * mean_rows * d * V / step_s / 1e12
    # the tensor cores' dense bf16 rate from unit counts and clocks: every SM completes 8192 bf16
    # FLOP per clock (one 128 x 256 x 16 tcgen05 MMA per 128 clocks), at the median SM clock
    # sampled during the timed region and at the maximum clock
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    arch_per_mhz = sms * 8192 * 1e6 / 1e12
    mhz_run = clk.get("sm_mhz") or None
    mhz_max = clk.get("sm_max_mhz") or peaks.get("sm_max_mhz", 2070.0)
    if cfg.dtype == "bf16":
        fwd_kernel = "FwdLseStoreEpi" if all_stored else "FwdLseEpi"
        roofline = {"kernel": f"umma_gemm_kernel<K,K,{fwd_kernel}> (fused forward; + O(N) finalize)",
                    "bound": "tensor", "achieved": achieved_tf, "peak": peak_tf, "unit": "TFLOP/s",
                    "frac": achieved_tf / peak_tf, "traffic": FWD_GEMM_TRAFFIC.get((cfg.name, fwd_kernel)),
                    "algorithmic_per_launch": f"2*N*d*V = {fwd_flops:.4g} FLOP",
                    "peak_note": f"bf16_tflops_sustained ({src}); kernel timed inside the step"}
    else:
        # f32 runs on the CUDA cores: 152 SMs x 128 FP32 lanes x 2 FLOP per FMA at the maximum clock
        alu_peak = 152 * 128 * 2 * peaks.get("sm_max_mhz", 2070.0) * 1e6 / 1e12
        roofline = {"kernel": "simt_gemm (f32 fused forward; + O(N) finalize)", "bound": "alu",
                    "achieved": achieved_tf, "peak": alu_peak, "unit": "TFLOP/s", "frac": achieved_tf / alu_peak,
                    "traffic": None, "algorithmic_per_launch": f"2*N*d*V = {fwd_flops:.4g} FLOP",
                    "peak_note": "FP32 FMA lanes x 2 x maximum SM clock (derived, not measured)"}
    # per step: sampler 1, packing 2, forward 3 (GEMM, finalize, loss reduction), backward 3 per
    # chunk (recompute, dH, dW; the backward splits a step's rows into ceil(N / chunk) chunks), or,
    # from the logit store, 3 (conversion to dZ, dH, dW over all rows)
    launches = sum(6 + (3 if st else 3 * (-(-n // args.chunk_rows))) for n, st in zip(step_rows, stored))
    out = {
        "metric": "prefix tokens/s (fused LM-head PS-PPO fwd+bwd, 1xGB300)",
        "value": rows_all / (ms_max * 1e-3),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms_max / args.steps,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": cfg.dtype,
        "data": "synthetic (seeded generator; random-init head)",
        "config": {"workload": describe(cfg),
                   "global_batch": cfg.B * world, "mean_prefix_rows": mean_rows, "sum_lengths": b.total_len,
                   "bwd_chunk_rows": args.chunk_rows,
                   "logits": (f"kept by the forward in the logit store ({store_rows} rows, "
                              f"{up.store.numel() / 1e9:.1f} GB), turned into dZ in place by the backward"
                              if all_stored else "recomputed by the backward" if not any(stored)
                              else f"store for steps of up to {store_rows} rows, recomputed above"),
                   "l2": f"inputs larger than L2 (hidden states {b.total_len * cfg.d * 2 / 1e9:.1f} GB, "
                         f"W {cfg.V * cfg.d * 2 / 1e9:.2f} GB, "
                         + (f"logit store {mean_rows * cfg.V * 2 / 1e9:.1f} GB per step)" if all_stored else
                            f"dZ chunk {args.chunk_rows * cfg.V * 2 / 1e9:.1f} GB)"),
                   "parallelism": ("data-parallel: prompt shards (global batch = ranks x P prompts, cutoffs "
                                   "by global completion index), dW and loss all-reduced over NCCL" if dp
                                   else "replicas" if world > 1 else "single GPU")},
        "pct_bf16_peak": {"credited_6NdV_tflops": credited_tf,
                          "of_measured_cublas_sustained": credited_tf / peak_tf,
                          "of_measured_cublas_burst": credited_tf / peaks["bf16_tflops"],
                          "measured_source": src,
                          "arch_tflops_at_run_clock": arch_per_mhz * mhz_run if mhz_run else None,
                          "of_arch_at_run_clock": credited_tf / (arch_per_mhz * mhz_run) if mhz_run else None,
                          "arch_tflops_at_max_clock": arch_per_mhz * mhz_max,
                          "of_arch_at_max_clock": credited_tf / (arch_per_mhz * mhz_max),
                          "of_nominal_2250": credited_tf / 2250.0,
                          "executed_tflops": credited_tf * executed / 6,
                          "executed_flops_per_row": f"{executed:.0f} d V",
                          "executed_of_arch_at_run_clock": (credited_tf * executed / 6) / (arch_per_mhz * mhz_run)
                          if mhz_run else None,
                          "arch_note": f"{sms} SMs x 8192 dense bf16 FLOP per SM per clock x SM clock (run: median "
                                       f"sampled under load; max: the clock limit); nominal 2250 TFLOP/s dense; "
                                       f"'measured_cublas' = MEASURED_PEAKS.json (torch.matmul 8192^3)"},
        "per_call_ms": {"sample": float(per[:, 0].mean()), "pack": float(per[:, 1].mean()),
                        "fwd": float(per[:, 2].mean()), "bwd": float(per[:, 3].mean()),
                        "exchange": float(per[:, 4].mean()),
                        "note": "pack includes its one host synchronisation (reading N); exchange = the "
                                "all-reduce of dW and the loss (data-parallel runs only)"},
        "pass_stats": pass_stats,
        "roofline": roofline,
        "roofline_backward": ({"kernels": ("logit-store conversion + dH + dW GEMMs (executed 4*N*d*V per step)"
                                           if all_stored else "recompute + dH + dW GEMMs (executed 6*N*d*V per step)"),
                               "bound": "tensor",
                               "achieved": (executed - 2) * mean_rows * d * V / (float(per[:, 3].mean()) * 1e-3) / 1e12,
                               "peak": peak_tf, "unit": "TFLOP/s",
                               "frac": (executed - 2) * mean_rows * d * V / (float(per[:, 3].mean()) * 1e-3) / 1e12
                               / peak_tf,
                               "traffic": None, "peak_note": "bf16_tflops_sustained"}
                              if cfg.dtype == "bf16" else None),
        "e2e": {"value": e_rows / (e_ms * 1e-3), "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": 8, "ms_per_step": e_ms / args.steps,
                "h2d_alone_ms": h2d_ms, "h2d_alone_gbs": h2d / (h2d_ms * 1e-3) / 1e9,
                "overlap": "next batch copied on a second stream during the current pass (InputStager)"},
        "full_control": full_control,
        **({"recompute_control": recompute_control} if recompute_control is not None else {}),
        **({"vocab_parallel": vocab_parallel} if vocab_parallel is not None else {}),
        "gpu_launches": launches,
        "clocks": clk,
    }
    if design is not None:
        out["design_stage"] = design
    if rank == 0 and not args.no_cpu_baseline:
        out["cpu_baseline"] = optional(cpu_baseline, cfg, b, args.cpu_rows)
    if world > 1:
        dist.destroy_process_group()
    if rank == 0:
        print(json.dumps(out))


def time_design_stage(cfg, b, dev, stream, reps=3):
    """The step upstream of the update pass (Algorithm 1, steps 7-9), timed on its own: one pass
    of the (old-policy) head over every rollout token for the score proxy and the top-16 next
    tokens, the reward-uncertainty proxy u_t per prompt and step, and the optimized design
    (closed form + PAV + cap, budget 128) into sampler masses."""
    import torch
    from paper_2606_29758_gb300 import CutoffDesign, DesignShape
    D = b.dev
    N = b.total_len
    cd = CutoffDesign(DesignShape(cfg.P, cfg.K, b.T_max, cfg.d, cfg.V, N, 16), device=dev)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(5)]
    t = []
    for r in range(reps + 1):
        ev[0].record(stream)
        cd.score(D["hid_full"], D["W"], D["tok_full"])
        ev[1].record(stream)
        cd.uncertainty(D["L"], D["R"])
        ev[2].record(stream)
        cd.design(D["L"], 128.0)
        ev[3].record(stream)
        cd.design(D["L"], 2048.0)
        ev[4].record(stream)
        torch.cuda.synchronize()
        if r > 0:
            t.append([ev[i].elapsed_time(ev[i + 1]) for i in range(4)])
    cd.check_status()
    saturated = int((cd.xi == 1.0).sum().item())
    pm, um, dm, dm2 = (float(x) for x in np.mean(np.array(t), axis=0))
    return {"rows": N, "proxy_topk_ms": pm, "uncertainty_ms": um, "design_ms": dm, "design_ms_budget_2048": dm2,
            "saturated_steps_budget_2048": saturated,
            "proxy_tflops": 2.0 * N * cfg.d * cfg.V / (pm * 1e-3) / 1e12,
            "note": "score proxy + top-16 over every rollout token (one head GEMM + epilogue), u_t, and the "
                    "optimized design (budget 128, and 2048, where the cap saturates long prefixes) per "
                    "prompt; not part of the timed step"}


def _oracle_prefix(cfg, b, step):
    """The oracle's cutoffs, advantages and packing indices for the whole batch (one step)."""
    from oracle.cutoffs import sample_cutoffs
    from oracle.pack import group_advantages, pack_prefixes
    H, n, w_tab = sample_cutoffs(b.q, b.L, cfg.K, cfg.seed, step)
    A = group_advantages(b.R, cfg.K, cfg.adv_mode)
    return pack_prefixes(b.L, n, cfg.K, w_tab, A, b.tok_full, b.oldlogp_full, None)


def _oracle_head(cfg, b, W64, pk, rows):
    """The oracle's head forward, dH and dW over the first `rows` packed rows of a step."""
    from oracle import lmhead
    from oracle.pipeline import widen
    s = np.arange(min(rows, pk["N"]))
    Hs = widen(cfg, b.hid_full[pk["src_row"][s]])
    f = lmhead.forward(Hs, W64, pk["tok"][s], pk["oldlogp"][s], pk["adv"][s], pk["w"][s], cfg.eps, cfg.loss_scale)
    lmhead.backward(Hs, W64, pk["tok"][s], f["lse"], f["coef"])
    return s.size


def _oracle_timing(cfg, b, W64, rows, step):
    """One step of the oracle, timed in parts: the whole batch's cutoffs, advantages and packing
    indices (in full), then the head on the first rows/2 and the first `rows` packed rows (whole
    128-row blocks of the oracle's head). A head call costs a fixed part (its V x d float64 dW
    accumulator, allocated and touched once per call) plus a part linear in the rows; the two sample
    sizes separate them, so a whole step is prefix + fixed + N x per-row."""
    t0 = time.perf_counter()
    pk = _oracle_prefix(cfg, b, step)
    t1 = time.perf_counter()
    small = _oracle_head(cfg, b, W64, pk, rows // 2)
    t2 = time.perf_counter()
    large = _oracle_head(cfg, b, W64, pk, rows)
    t3 = time.perf_counter()
    return {"N": pk["N"], "prefix_s": t1 - t0, "rows": (small, large), "head_s": (t2 - t1, t3 - t2)}


def _oracle_summary(ts):
    N = float(np.mean([t["N"] for t in ts]))
    prefix_s = float(np.mean([t["prefix_s"] for t in ts]))
    d_rows = sum(t["rows"][1] - t["rows"][0] for t in ts)
    d_s = sum(t["head_s"][1] - t["head_s"][0] for t in ts)
    if d_rows > 0 and d_s > 0:
        per_row = d_s / d_rows
        fixed = max(0.0, float(np.mean([t["head_s"][1] - t["rows"][1] * per_row for t in ts])))
    else:   # samples too small to separate the two parts (timing noise): all of it per row
        per_row = sum(t["head_s"][1] for t in ts) / max(1, sum(t["rows"][1] for t in ts))
        fixed = 0.0
    step_s = prefix_s + fixed + N * per_row
    return {"value": N / step_s, "unit": "tokens/s", "head_rows_per_s": 1.0 / per_row, "head_fixed_s": fixed,
            "prefix_s_per_step": prefix_s, "extrapolated_step_s": step_s, "mean_prefix_rows": N}


def cpu_baseline(cfg, b, rows):
    from oracle.pipeline import widen
    W64 = widen(cfg, b.W)
    t = _oracle_timing(cfg, b, W64, rows, 0)
    out = _oracle_summary([t])
    out.update({"cores": os.cpu_count(), "kind": "oracle",
                "sample": f"one {cfg.name} step: cutoffs, advantages and packing indices of the whole batch "
                          f"({t['prefix_s']:.2f} s), then the f64 head forward + dH + dW over {t['rows'][0]} and "
                          f"{t['rows'][1]} packed rows ({t['head_s'][0]:.1f} + {t['head_s'][1]:.1f} s): a fixed "
                          f"{out['head_fixed_s']:.2f} s per head call plus {1e3 / out['head_rows_per_s']:.1f} ms per "
                          f"row; value = the step's packed rows / (prefix + fixed + rows x per-row), extrapolated"})
    return out


def run_reference(args):
    from synthetic import get_config, make_batch
    from oracle.pipeline import widen
    world, rank, _ = _dist()
    if rank != 0:
        return
    cfg = get_config(args.config)
    dev = None
    try:
        import torch
        if torch.cuda.is_available():
            dev = "cuda:0"
    except Exception:
        pass
    b = make_batch(cfg, device=dev)   # the old log-probs need the full head; on the GPU when present
    W64 = widen(cfg, b.W)
    for i in range(args.warmup):
        _oracle_timing(cfg, b, W64, args.ref_rows, 1000 + i)
    t0 = time.perf_counter()
    ts = [_oracle_timing(cfg, b, W64, args.ref_rows, i) for i in range(args.steps)]
    dt = time.perf_counter() - t0
    summ = _oracle_summary(ts)
    v = summ["value"]
    print(json.dumps({
        "impl": "reference", "metric": "prefix tokens/s (fused LM-head PS-PPO fwd+bwd, 1xGB300)",
        "value": v, "unit": "tokens/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": summ["extrapolated_step_s"] * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded generator; random-init head)",
        "config": {"workload": describe(cfg), "sample_rows_per_step": args.ref_rows},
        "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
                         "head_rows_per_s": summ["head_rows_per_s"], "head_fixed_s": summ["head_fixed_s"],
                         "prefix_s_per_step": summ["prefix_s_per_step"],
                         "sample": f"{args.steps} steps, each: cutoffs, advantages and packing indices of the "
                                   f"whole batch in full, then the f64 head forward + dH + dW over "
                                   f"{args.ref_rows // 2} and {args.ref_rows} packed rows ({dt:.1f} s in all); "
                                   f"value and ms_per_step = one whole step extrapolated: prefix time + the head's "
                                   f"fixed cost per call + N x its per-row cost"},
        "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


def run_torch(args):
    """Context arm: the same step with the head in eager PyTorch (cuBLAS GEMMs, logits
    materialised per row chunk, autograd for dH and dW); sampling and packing through the library."""
    import torch
    from paper_2606_29758_gb300 import PassShape, UpdatePass
    from synthetic import get_config, make_batch
    world, rank, local = _dist()
    if rank != 0:
        return
    torch.cuda.set_device(local)
    dev = f"cuda:{local}"
    cfg = get_config(args.config)
    b = make_batch(cfg, device=dev)
    D = b.dev
    # the library's backward workspace is not used here: keep it at its minimum (128 rows)
    up = UpdatePass(PassShape(cfg.P, cfg.K, b.T_max, cfg.d, cfg.V, b.total_len, torch.bfloat16, 128),
                    device=dev, eps=cfg.eps, loss_scale=cfg.loss_scale)
    W = D["W"].clone().requires_grad_(True)
    chunk = args.torch_chunk

    def step(i):
        up.sample(D["q"], D["L"], cfg.seed, i)
        n = up.pack(D["L"], D["R"], D["tok_full"], D["oldlogp_full"], D["hid_full"])
        W.grad = None
        for r0 in range(0, n, chunk):
            r1 = min(n, r0 + chunk)
            h = up.hid[r0:r1].detach().requires_grad_(True)
            z = (h @ W.t()).float()
            lp = z.gather(1, up.tok[r0:r1, None].long())[:, 0] - torch.logsumexp(z, dim=1)
            r = torch.exp(lp - up.oldlogp[r0:r1])
            A = up.adv[r0:r1]
            sur = torch.minimum(r * A, torch.clamp(r, 1 - cfg.eps, 1 + cfg.eps) * A)
            (-(cfg.loss_scale * up.w[r0:r1] * sur).sum()).backward()
            up.dH[r0:r1] = h.grad
        return n

    for i in range(args.warmup):
        step(1000 + i)
    torch.cuda.synchronize()
    torch.cuda.reset_peak_memory_stats()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record()
    rows = sum(step(i) for i in range(args.steps))
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    print(json.dumps({
        "impl": "torch-eager", "metric": "prefix tokens/s (fused LM-head PS-PPO fwd+bwd, 1xGB300)",
        "value": rows / (ms * 1e-3), "unit": "tokens/s", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms / args.steps, "higher_is_better": True, "dtype": "bf16",
        "config": {"workload": describe(cfg), "logit_chunk_rows": chunk},
        "peak_device_memory_gb": torch.cuda.max_memory_allocated() / 1e9,
        "note": "context only: the head in eager PyTorch (cuBLAS GEMMs, logits materialised per chunk, "
                "autograd); cutoffs and packing through the library"}))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference", "torch"], default="ours")
    ap.add_argument("--torch-chunk", type=int, default=16384, help="rows per logit chunk of --impl torch")
    ap.add_argument("--config", default=WORKLOAD)
    ap.add_argument("--chunk-rows", type=int, default=65536)
    ap.add_argument("--logits", choices=["recompute", "store"], default="store",
                    help="keep the logits from the forward (logit store, where the device memory holds it) or "
                         "recompute them in the backward")
    ap.add_argument("--cpu-rows", type=int, default=256)
    # the head is timed on ref_rows/2 and ref_rows packed rows, whole 128-row blocks of the oracle's
    # head (its dW update touches all of V x d once per block), separating its per-call and per-row cost
    ap.add_argument("--ref-rows", type=int, default=256)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-design", action="store_true", help="skip timing the cutoff-design stage")
    ap.add_argument("--vocab-shards", type=int, default=0,
                    help="also time the step with the head split into this many vocabulary shards (context)")
    ap.add_argument("--replicas", action="store_true",
                    help="with several ranks: independent replicas, no exchange of dW")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    elif args.impl == "torch":
        run_torch(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
