"""Throughput of the BGPO masked-diffusion ELBO hot path on GB300.

One step = Algorithm 1's inner loops over one batch: for every MC sample j,
sample_mask -> elbo_fwd -> bound_coeffs -> elbo_bwd_accumulate, through the C ABI
of include/bgpo.h (all arithmetic in the library's CUDA kernels). Workload:
LLaDA-8B-shaped LM head (H=4096, V=126464), 16 responses of 512 tokens after a
256-token prompt, n_t=16 stratified MC samples, on-policy (old = current).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

Prints ONE JSON line (rank 0). `value` = masked tokens/s over all ranks with
inputs resident in HBM; `e2e` = the same through host (pinned) buffers with the
host<->device copies inside the timed region; `roofline` = the dominant kernel's
algorithmic tensor FLOP/s against the measured bf16 peak; `cpu_baseline` = the
fp64 oracle on a bounded sample of the same workload on the host cores.
`--impl reference` times that oracle alone (the reference arm of this tier).

The step runs with BGPO_FLAG_PAIR_DW (MC samples 2k and 2k + 1 share one dW
GEMM; the loop above is exactly the call order that flag expects) unless
`--no-pair-dw` is given. `unpaired` = the same step without it (the library's
default flags: the backward walks the vocabulary in chunks of at most 32,768
columns, so its dL/dz buffer holds one chunk); `unpaired_whole_vocab` = the
unpaired step with the whole vocabulary as one chunk; `keep_logits` = the
paired step with BGPO_FLAG_KEEP_LOGITS too (the forward keeps its fp32 logits,
the backward reads them instead of recomputing them).

Under torchrun (N > 1) every rank owns B responses of an N * B batch and each
step ends with the one data-parallel exchange, the sum of dW over the ranks
(paper_2510_11683_gb300.dp.allreduce_dw, NCCL), inside the timed region.
"""
import argparse
import hashlib
import json
import os
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = "llada8b_r512_onpolicy"
METRIC = "masked tokens/s (fwd+bwd)"
UNIT = "tokens/s"

# dram__bytes_read.sum + dram__bytes_write.sum per launch of each GEMM kind,
# the mean over every launch of one bench step of `workload` (dW paired, the
# logits recomputed: the headline leg), from one ncu capture of those launches
# (a one-pass metric set, caches cold before each launch). Valid for that
# workload while the GEMM sources hash to `sha`; otherwise the line reports
# traffic as null.
TRAFFIC = {
    "sha": "981f980e3a7dad317219b89f4aa070d106cc6dba692a8370f6e7e2c06829d45a",
    "workload": "llada8b_r512_onpolicy",
    "bytes_per_launch": {"lmhead_fwd_lse": 1.561e9, "lmhead_dz": 3.275e9, "dx_gemm": 4.363e9,
                         "dw_gemm": 14.406e9},
    "source": "ncu over the 56 GEMM launches of one bench step (llada8b_r512_onpolicy, dW paired), "
              "mean per launch",
}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--workload", default=WORKLOAD)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-sweep", action="store_true")
    ap.add_argument("--no-keep-logits", action="store_true",
                    help="skip the timed leg with BGPO_FLAG_KEEP_LOGITS")
    ap.add_argument("--no-pair-dw", action="store_true",
                    help="time the step without BGPO_FLAG_PAIR_DW (and skip the unpaired leg)")
    ap.add_argument("--no-whole-vocab", action="store_true",
                    help="skip the unpaired leg with the whole vocabulary as one chunk")
    ap.add_argument("--grad-variance", action="store_true",
                    help="run the Sec. 4.3 gradient std / bias vs n_t study instead")
    ap.add_argument("--profile-sample", type=int, default=None, metavar="J",
                    help="run MC sample J's path once (mask, forward, coefficients, backward; "
                         "with dW paired and J odd, sample J - 1 first) and exit: a short "
                         "process whose kernels ncu can capture after few launches")
    ap.add_argument("--vocab-chunk", type=int, default=0,
                    help="bgpo_problem.vocab_chunk for --profile-sample (0 = default)")
    ap.add_argument("--keep", action="store_true",
                    help="BGPO_FLAG_KEEP_LOGITS for --profile-sample")
    return ap.parse_args()


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return dict(bf16=float(d["bf16_tflops"]), bf16_sustained=float(d["bf16_tflops_sustained"]),
                    hbm=float(d["hbm_gbs"]), source="measured")
    return dict(bf16=1900.0, bf16_sustained=1700.0, hbm=6800.0, source="fallback")


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms while running."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except OSError:
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
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for name, val in zip(names, parts[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": max(smax),
                "samples": len(sm), "reasons": sorted(reasons)}


# ----------------------------------------------------------------------------------
# CPU baseline / reference arm: the fp64 oracle as it stands, on a bounded sample
# ----------------------------------------------------------------------------------

def oracle_sample(wl, inp_cpu, budget_s=12.0, max_seqs=4):
    """Times the oracle's per-sample path (Eq. 4 forward, Eq. 10/13 bound, gradients)
    for MC sample j = n_t/2 on sequences 0, 1, ... until `budget_s` has passed.
    Returns (masked rows processed, seconds, description)."""
    from oracle import bgpo_oracle as O
    from tests.harness import to64

    X = to64(inp_cpu["X"])
    W = to64(inp_cpu["W"])
    Y = to64(inp_cpu["Y"])
    j = wl.n_t // 2
    _, _, t, mask = O.sample_t_mask(wl.seed, wl.B, wl.R, j, wl.n_t, wl.t_mode)
    rows = 0
    seqs = 0
    t0 = time.perf_counter()
    for b in range(min(wl.B, max_seqs)):
        sub = np.zeros_like(mask)
        sub[b] = mask[b]
        ell = O.elbo_term(X, W, Y, wl.P, sub, t)
        _, _, coef = O.bound_coeffs(ell, ell, np.ones(wl.B), wl.n_t, 1.0 / wl.G)
        O.elbo_term_grads(X, W, Y, wl.P, sub, t, coef)
        rows += int(mask[b].sum())
        seqs += 1
        if time.perf_counter() - t0 > budget_s:
            break
    dt = time.perf_counter() - t0
    desc = (f"oracle fp64 (numpy, BLAS on all host cores): MC sample j={j} of sequences "
            f"0..{seqs - 1} ({rows} masked rows, full V={wl.V}, H={wl.H}): forward, bound "
            f"coefficients and gradients")
    return rows, dt, desc


def run_reference(args, wl):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    from synth import make_inputs
    inp = make_inputs(wl)
    for _ in range(args.warmup):
        oracle_sample(wl, inp, budget_s=2.0, max_seqs=1)
    tot_rows, tot_s = 0, 0.0
    desc = ""
    for _ in range(args.steps):
        rows, dt, desc = oracle_sample(wl, inp, budget_s=4.0, max_seqs=1)
        tot_rows += rows
        tot_s += dt
    value = tot_rows / tot_s
    cores = os.cpu_count()
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot_s / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": config_of(wl),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": desc},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


L2_BYTES = 129e6


def config_of(wl):
    head = {(4096, 126464): "LLaDA-8B-shaped LM head",
            (3584, 152064): "Dream-7B-shaped LM head"}.get((wl.H, wl.V), "LM head")
    w_bytes = 2.0 * wl.H * wl.V
    l2 = (f"inputs larger than L2 (W alone is {w_bytes / 1e9:.2f} GB > 129 MB); no flush"
          if w_bytes > L2_BYTES else
          f"inputs fit in L2 (W is {w_bytes / 1e6:.2f} MB); no flush: a launch-bound case")
    return {"workload": f"{wl.name}: {head} H={wl.H} V={wl.V}, {wl.B} responses "
                        f"x (prompt {wl.P} + response {wl.R}), n_t={wl.n_t} "
                        f"{'stratified' if wl.t_mode else 'iid'} t, G={wl.G}, "
                        f"{'on-policy' if wl.eps_std == 0 else 'off-policy'}",
            "B": wl.B, "P": wl.P, "R": wl.R, "H": wl.H, "V": wl.V, "n_t": wl.n_t, "G": wl.G,
            "l2": l2}


# ----------------------------------------------------------------------------------
# native arm
# ----------------------------------------------------------------------------------

def aggregate_ranks(ms_local, tokens_local):
    """Whole-job figures of a data-parallel run: the slowest rank's ms per step
    and the masked tokens of all ranks (torch.distributed must be initialised
    when the world is larger than one)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return ms_local, tokens_local
    dev = torch.device("cuda", torch.cuda.current_device()) \
        if dist.get_backend() == "nccl" else torch.device("cpu")
    t = torch.tensor([ms_local], dtype=torch.float64, device=dev)
    n = torch.tensor([tokens_local], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(n, op=dist.ReduceOp.SUM)
    return float(t.item()), int(n.item())


def shard_of(wl, rank, world):
    """(data workload, b_offset) of `rank`: every rank owns its own B responses,
    which are sequences [rank * B, (rank + 1) * B) of a world * B batch; draws use
    the batch seed and the global sequence index, data draws a per-rank seed."""
    if world == 1:
        return wl, 0
    return wl.with_(seed=wl.seed + 7919 * rank), rank * wl.B


def kernel_sha():
    """sha256 of the GEMM kernel sources (k_gemm.cu and the headers it inlines)."""
    h = hashlib.sha256()
    for name in ("k_gemm.cu", "bgpo_device.cuh", "bgpo_plan.h"):
        with open(os.path.join(ROOT, "paper_2510_11683_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def main():
    args = parse()
    from synth import CONFIGS
    wl = CONFIGS[args.workload]
    if args.impl == "reference":
        run_reference(args, wl)
        return
    if args.grad_variance:
        run_grad_variance(args, CONFIGS["llada8b_sweep"] if args.workload == WORKLOAD else wl)
        return
    if args.profile_sample is not None:
        run_profile_sample(args, wl)
        return

    import torch
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        # NCCL's own start-up lines (ranks, devices) stay in the log
        os.environ.setdefault("NCCL_DEBUG", "INFO")
        os.environ.setdefault("NCCL_DEBUG_SUBSYS", "INIT")
    # each rank drives the GPU of its local rank; select it before NCCL binds
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)

    import paper_2510_11683_gb300 as bg
    from paper_2510_11683_gb300 import build as B
    from paper_2510_11683_gb300.dp import allreduce_dw
    if not os.path.exists(B.LIB_PATH):
        B.build()
    from synth import make_inputs

    # weak scaling: every rank owns B responses of a world * B batch; the data
    # path has no collective, and each step ends with the sum of dW over ranks
    wl_data, b_offset = shard_of(wl, rank, world)
    inp_cpu = make_inputs(wl_data)
    inp = {k: (v.to(dev) if v is not None else None) for k, v in inp_cpu.items()}
    X, W, Y = inp["X"], inp["W"], inp["Y"]
    n_t, Bsz = wl.n_t, wl.B

    pair = not args.no_pair_dw
    prob = bg.problem_from(wl, b_offset=b_offset, pair_dw=pair)
    ws = bg.alloc_workspace(prob, dev)
    bg.clear_device_error(ws)
    A = torch.empty(Bsz, dtype=torch.float32, device=dev)
    if inp["A"] is not None:
        A.copy_(inp["A"])
    else:
        bg.group_advantage(prob, inp["rewards"], A)

    # old-policy pass (outside the timed step, forward only): l_old on the same
    # draws (Eq. 10)
    ell_old = torch.empty((n_t, Bsz), dtype=torch.float32, device=dev)
    masks = torch.empty((n_t, Bsz, wl.R), dtype=torch.uint8, device=dev)
    for j in range(n_t):
        bg.sample_mask(prob, j, ws, None, masks[j])
        bg.elbo_fwd(prob, j, X, W, Y, ws, ell_old[j])
    ell_old += inp["eps"].T.to(dev)
    masked_per_step = int(masks.sum().item())
    rows_per_sample = masks.reshape(n_t, -1).sum(dim=1).tolist()

    ell = torch.empty((n_t, Bsz), dtype=torch.float32, device=dev)
    coef = torch.empty((n_t, Bsz), dtype=torch.float32, device=dev)
    g = torch.empty((n_t, Bsz), dtype=torch.float32, device=dev)
    dX = torch.zeros((Bsz, wl.R, wl.H), dtype=torch.float32, device=dev)
    dW = torch.zeros((wl.V, wl.H), dtype=torch.float32, device=dev)

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    def timed_leg(keep, pair_dw, ws_, sample_clocks, vocab_chunk=0):
        """W warm-up and K timed steps of one mode; per-kernel times from the trace."""
        def step(p):
            for j in range(n_t):
                bg.sample_mask(p, j, ws_)
                bg.elbo_fwd(p, j, X, W, Y, ws_, ell[j])
                bg.bound_coeffs(p, j, ell[j], ell_old[j], A, coef[j], g[j], ws_)
                bg.elbo_bwd_accumulate(p, j, X, W, Y, coef[j], ws_, dX, dW)
            allreduce_dw(dW)      # the data-parallel exchange (a no-op on one rank)

        for _ in range(args.warmup):
            step(bg.problem_from(wl, b_offset=b_offset, keep_logits=keep, pair_dw=pair_dw,
                                 vocab_chunk=vocab_chunk))
        torch.cuda.synchronize()
        chunks = -(-wl.V // (vocab_chunk or 32768))     # at most this many vocabulary chunks
        trace = bg.Trace(args.steps * n_t * (8 + 3 * chunks) + 16)
        prob_t = bg.problem_from(wl, trace=trace, b_offset=b_offset, keep_logits=keep,
                                 pair_dw=pair_dw, vocab_chunk=vocab_chunk)
        clocks = ClockSampler(torch.cuda.current_device() if world == 1 else local)
        stream = torch.cuda.current_stream()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        barrier()
        torch.cuda.synchronize()
        if sample_clocks:
            clocks.start()
            time.sleep(0.3)
        e0.record(stream)
        for _ in range(args.steps):
            step(prob_t)
        e1.record(stream)
        torch.cuda.synchronize()
        barrier()
        clock_info = clocks.stop() if sample_clocks else None
        code, where = bg.get_device_error(ws_)
        if code != 0:
            raise RuntimeError(f"device error {code} at {where}")
        recs = trace.records()
        per_kernel = {}
        for name, kms in recs:
            d = per_kernel.setdefault(name, [0, 0.0])
            d[0] += 1
            d[1] += kms
        trace.close()
        return e0.elapsed_time(e1) / args.steps, per_kernel, clock_info, len(recs)

    peaks = load_peaks()
    H, V = wl.H, wl.V
    gemm_flops_per_step = 2.0 * H * V * masked_per_step   # each GEMM kind of the step

    def rooflines(per_kernel, headline_mode):
        """Dominant GEMM against the sustained bf16 peak; the dz pass (if any) against HBM.
        `headline_mode`: the leg runs the bench step (dW paired, logits recomputed),
        the mode TRAFFIC was measured in."""
        gemm_kernels = [k for k in ("lmhead_fwd_lse", "lmhead_dz", "dx_gemm", "dw_gemm")
                        if k in per_kernel]
        dom = max(gemm_kernels, key=lambda k: per_kernel[k][1])
        dom_launches, dom_ms = per_kernel[dom]
        dom_flops_per_launch = gemm_flops_per_step * args.steps / dom_launches
        dom_avg_s = dom_ms / dom_launches / 1e3
        achieved = dom_flops_per_launch / dom_avg_s / 1e12
        traffic = None
        if (headline_mode and args.workload == TRAFFIC["workload"] and world == 1
                and TRAFFIC["sha"] == kernel_sha()):
            traffic = TRAFFIC["bytes_per_launch"].get(dom)
        roof = {"bound": "tensor", "achieved": achieved, "peak": peaks["bf16_sustained"],
                "unit": "TFLOP/s", "frac": achieved / peaks["bf16_sustained"], "traffic": traffic,
                "traffic_source": TRAFFIC["source"] if traffic is not None else None,
                "kernel": dom, "peak_kind": f"bf16 sustained ({peaks['source']})",
                "flops_per_launch": dom_flops_per_launch, "avg_launch_ms": dom_avg_s * 1e3}
        # dL/dz from kept logits: reads 4 V and writes 2 V bytes per masked row
        hbm_pass = None
        if "dz_from_logits" in per_kernel:
            n_dz, dz_ms = per_kernel["dz_from_logits"]
            dz_bytes = 6.0 * V * masked_per_step * args.steps / n_dz
            dz_gbs = dz_bytes / (dz_ms / n_dz / 1e3) / 1e9
            hbm_pass = {"kernel": "dz_from_logits", "bound": "hbm", "achieved": dz_gbs,
                        "peak": peaks["hbm"], "unit": "GB/s", "frac": dz_gbs / peaks["hbm"],
                        "bytes_per_launch": dz_bytes, "avg_launch_ms": dz_ms / n_dz,
                        "peak_kind": f"HBM copy ({peaks['source']})"}
        return roof, hbm_pass, len(gemm_kernels)

    # headline: logits recomputed in the backward, never stored; dW paired
    ms_local, per_kernel, clock_info, gpu_launches = timed_leg(False, pair, ws, True)
    ms, masked_all = aggregate_ranks(ms_local, masked_per_step)
    roofline, _, n_gemm = rooflines(per_kernel, pair)
    value = masked_all / (ms / 1e3)
    exec_tflops = n_gemm * gemm_flops_per_step / (ms / 1e3) / 1e12
    useful_tflops = 3 * gemm_flops_per_step / (ms / 1e3) / 1e12   # fwd, dX, dW

    out = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic (seeded; shapes of the paper's "
        "LLaDA-8B head, response 512, n_t=16)", "config": config_of(wl),
        "roofline": roofline, "gpu_launches": gpu_launches, "clocks": clock_info,
        "library_flags": ["BGPO_FLAG_PAIR_DW"] if pair else [],
        "mc_samples_per_s": Bsz * n_t * world / (ms / 1e3),
        "masked_rows_per_step": masked_per_step, "masked_rows_per_sample": rows_per_sample,
        "step_tensor_tflops_executed": exec_tflops,
        "step_frac_of_bf16_peak_executed": exec_tflops / peaks["bf16"],
        "step_frac_of_bf16_peak_useful": useful_tflops / peaks["bf16"],
        "per_kernel_ms_per_step": {k: v[1] / args.steps for k, v in per_kernel.items()},
        "peak_mem_bytes": torch.cuda.max_memory_allocated(dev),
        "workspace_bytes": ws.numel(),
    }
    if rank == 0:
        print(f"[bench] {ms:.2f} ms/step, {value:.4g} tok/s, dominant {roofline['kernel']} "
              f"{roofline['achieved']:.1f} TFLOP/s, per kernel ms/step: "
              f"{ {k: round(v[1] / args.steps, 3) for k, v in per_kernel.items()} }",
              file=sys.stderr, flush=True)

    # the same step with the library's default flags (a dW GEMM per sample and
    # vocabulary chunk, dL/dz one chunk at a time), and with the whole
    # vocabulary as one chunk
    legs = [("unpaired", 0)] + ([] if args.no_whole_vocab else [("unpaired_whole_vocab", 1 << 24)])
    for leg, chunk in (legs if rank == 0 and world == 1 and pair else []):
        ws_u = bg.alloc_workspace(bg.problem_from(wl, b_offset=b_offset, vocab_chunk=chunk), dev)
        u_ms, u_per_kernel, _, u_launches = timed_leg(False, False, ws_u, False, chunk)
        u_roof, _, _ = rooflines(u_per_kernel, False)
        out[leg] = {
            "value": masked_per_step / (u_ms / 1e3), "unit": UNIT, "ms_per_step": u_ms,
            "gpu_launches": u_launches, "roofline": u_roof, "vocab_chunk": chunk,
            "workspace_bytes": ws_u.numel(),
            "per_kernel_ms_per_step": {k: v[1] / args.steps for k, v in u_per_kernel.items()}}
        print(f"[bench] {leg}: {u_ms:.2f} ms/step, {masked_per_step / (u_ms / 1e3):.4g} tok/s, "
              f"per kernel ms/step: "
              f"{ {k: round(v[1] / args.steps, 3) for k, v in u_per_kernel.items()} }",
              file=sys.stderr, flush=True)
        del ws_u
        torch.cuda.empty_cache()

    # the same step with BGPO_FLAG_KEEP_LOGITS (the forward keeps its fp32 logits,
    # the backward forms dL/dz from them in one HBM pass instead of a fourth GEMM)
    if rank == 0 and world == 1 and not args.no_keep_logits:
        del ws
        torch.cuda.empty_cache()
        torch.cuda.reset_peak_memory_stats(dev)
        ws_keep = bg.alloc_workspace(
            bg.problem_from(wl, b_offset=b_offset, keep_logits=True, pair_dw=pair), dev)
        k_ms, k_per_kernel, _, k_launches = timed_leg(True, pair, ws_keep, False)
        k_roof, k_hbm, _ = rooflines(k_per_kernel, False)
        out["keep_logits"] = {
            "value": masked_per_step / (k_ms / 1e3), "unit": UNIT, "ms_per_step": k_ms,
            "gpu_launches": k_launches, "roofline": k_roof, "roofline_hbm_pass": k_hbm,
            "step_frac_of_bf16_peak_executed":
                3 * gemm_flops_per_step / (k_ms / 1e3) / 1e12 / peaks["bf16"],
            "per_kernel_ms_per_step": {k: v[1] / args.steps for k, v in k_per_kernel.items()},
            "peak_mem_bytes": torch.cuda.max_memory_allocated(dev),
            "workspace_bytes": ws_keep.numel()}
        print(f"[bench] keep_logits: {k_ms:.2f} ms/step, {masked_per_step / (k_ms / 1e3):.4g} tok/s, "
              f"per kernel ms/step: "
              f"{ {k: round(v[1] / args.steps, 3) for k, v in k_per_kernel.items()} }",
              file=sys.stderr, flush=True)
        del ws_keep
        torch.cuda.empty_cache()

    if not args.no_e2e:
        # every rank times its own shard end to end; whole job = all ranks'
        # tokens over the slowest rank's time
        e = e2e_leg(bg, wl, inp_cpu, ell_old.cpu(), masked_per_step, args, dev, b_offset, barrier,
                    pair)
        e_ms, e_tokens = aggregate_ranks(e["ms_per_step"], masked_per_step)
        e.update(value=e_tokens / (e_ms / 1e3), ms_per_step=e_ms,
                 h2d_bytes_per_step=e["h2d_bytes_per_step"] * world,
                 d2h_bytes_per_step=e["d2h_bytes_per_step"] * world)
        out["e2e"] = e

    if rank == 0 and world == 1 and not args.no_sweep:
        del dX, dW
        torch.cuda.empty_cache()
        out["nt_sweep"] = nt_sweep(bg, dev, pair)

    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        rows, dt, desc = oracle_sample(wl, inp_cpu)
        out["cpu_baseline"] = {"value": rows / dt, "unit": UNIT, "cores": os.cpu_count(),
                               "kind": "oracle", "sample": desc, "seconds": dt}

    if rank == 0:
        print(json.dumps(out), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def e2e_leg(bg, wl, inp_cpu, ell_old_cpu, masked_per_step, args, dev, b_offset=0,
            barrier=lambda: None, pair=False):
    """Same step through host buffers: every step copies its inputs (X, W, Y,
    rewards or A, l_old) from pinned host memory and copies its results (l and
    g) back to pinned host memory, where the host reads them. Input copies run
    on a second stream into the other of two device buffer sets, so step k+1's
    inputs travel while step k computes; the host reads step k - 1's results
    while step k runs, as a training loop that logs the previous step's loss
    does. All copies and reads lie inside the timed region."""
    import torch
    from paper_2510_11683_gb300.dp import allreduce_dw
    n_t, Bsz = wl.n_t, wl.B
    host = {
        "X": inp_cpu["X"].pin_memory(), "W": inp_cpu["W"].pin_memory(),
        "Y": inp_cpu["Y"].pin_memory(), "old": ell_old_cpu.contiguous().pin_memory(),
    }
    adv_key = "A" if inp_cpu["A"] is not None else "rewards"
    host["adv"] = inp_cpu[adv_key].pin_memory()
    bufs = [{k: torch.empty_like(v, device=dev) for k, v in host.items()} for _ in range(2)]
    out_ell = [torch.empty((n_t, Bsz), dtype=torch.float32).pin_memory() for _ in range(2)]
    out_g = [torch.empty((n_t, Bsz), dtype=torch.float32).pin_memory() for _ in range(2)]
    prob = bg.problem_from(wl, b_offset=b_offset, pair_dw=pair)
    ws = bg.alloc_workspace(prob, dev)
    A = torch.empty(Bsz, dtype=torch.float32, device=dev)
    ell = torch.empty((n_t, Bsz), dtype=torch.float32, device=dev)
    coef = torch.empty_like(ell)
    g = torch.empty_like(ell)
    dX = torch.zeros((Bsz, wl.R, wl.H), dtype=torch.float32, device=dev)
    dW = torch.zeros((wl.V, wl.H), dtype=torch.float32, device=dev)
    h2d = sum(v.numel() * v.element_size() for v in host.values())
    d2h = out_ell[0].numel() * 4 + out_g[0].numel() * 4
    compute = torch.cuda.current_stream()
    copy = torch.cuda.Stream(device=dev)
    copied = [torch.cuda.Event(), torch.cuda.Event()]
    consumed = [torch.cuda.Event(), torch.cuda.Event()]
    ready = [torch.cuda.Event(), torch.cuda.Event()]   # a step's results are on the host
    seen = []                                          # what the host read, per step

    def issue_copy(k):
        slot = k % 2
        with torch.cuda.stream(copy):
            copy.wait_event(consumed[slot])      # the step that last used this slot is done
            for name in host:
                bufs[slot][name].copy_(host[name], non_blocking=True)
            copied[slot].record(copy)

    def compute_step(k):
        slot = k % 2
        b = bufs[slot]
        compute.wait_event(copied[slot])
        if adv_key == "A":
            A.copy_(b["adv"])
        else:
            bg.group_advantage(prob, b["adv"], A)
        for j in range(n_t):
            bg.sample_mask(prob, j, ws)
            bg.elbo_fwd(prob, j, b["X"], b["W"], b["Y"], ws, ell[j])
            bg.bound_coeffs(prob, j, ell[j], b["old"][j], A, coef[j], g[j], ws)
            bg.elbo_bwd_accumulate(prob, j, b["X"], b["W"], b["Y"], coef[j], ws, dX, dW)
        allreduce_dw(dW)          # the data-parallel exchange (a no-op on one rank)
        consumed[slot].record(compute)
        out_ell[slot].copy_(ell, non_blocking=True)
        out_g[slot].copy_(g, non_blocking=True)
        ready[slot].record(compute)

    def read(k):
        ready[k % 2].synchronize()
        seen.append((float(out_ell[k % 2].sum()), float(out_g[k % 2].sum())))

    def run(steps):
        issue_copy(0)
        for k in range(steps):
            if k + 1 < steps:
                issue_copy(k + 1)
            compute_step(k)
            if k > 0:
                read(k - 1)          # step k - 1's results, while step k runs
        read(steps - 1)
    for e in consumed:
        e.record(compute)
    run(max(1, min(args.warmup, 2)))
    torch.cuda.synchronize()
    steps = max(2, args.steps)   # the first step's copies are exposed once per run
    barrier()
    t0 = time.perf_counter()
    run(steps)
    torch.cuda.synchronize()
    dt = (time.perf_counter() - t0) / steps
    barrier()
    return {"value": masked_per_step / dt, "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "ms_per_step": dt * 1e3, "steps": steps,
            "pipelining": "inputs of step k+1 copied on a second stream during step k; the host "
                          "reads step k-1's results during step k",
            "results_finite": bool(all(np.isfinite(v) for pair in seen for v in pair))}


def run_profile_sample(args, wl):
    """One MC sample's path through the C ABI with as few launches as possible
    before it: inputs, advantages, then mask, forward, coefficients (on-policy,
    d = 0) and backward of sample J (of J - 1 and J when dW is paired and J is
    odd). Prints the masked rows and the device error word per sample."""
    import torch
    import paper_2510_11683_gb300 as bg
    from paper_2510_11683_gb300 import build as B
    from synth import make_inputs
    if not os.path.exists(B.LIB_PATH):
        B.build()
    pair = not args.no_pair_dw
    inp = make_inputs(wl, device="cuda")
    X, W, Y = inp["X"], inp["W"], inp["Y"]
    p = bg.problem_from(wl, pair_dw=pair, keep_logits=args.keep, vocab_chunk=args.vocab_chunk)
    ws = bg.alloc_workspace(p)
    A = torch.empty(wl.B, dtype=torch.float32, device="cuda")
    if inp["A"] is not None:
        A.copy_(inp["A"])
    else:
        bg.group_advantage(p, inp["rewards"], A)
    ell = torch.empty(wl.B, dtype=torch.float32, device="cuda")
    coef = torch.empty_like(ell)
    dX = torch.zeros((wl.B, wl.R, wl.H), dtype=torch.float32, device="cuda")
    dW = torch.zeros((wl.V, wl.H), dtype=torch.float32, device="cuda")
    m = torch.empty((wl.B, wl.R), dtype=torch.uint8, device="cuda")
    j = args.profile_sample
    for jj in ([j - 1, j] if pair and j % 2 == 1 else [j]):
        bg.sample_mask(p, jj, ws, None, m)
        bg.elbo_fwd(p, jj, X, W, Y, ws, ell)
        bg.bound_coeffs(p, jj, ell, ell, A, coef, None, ws)
        bg.elbo_bwd_accumulate(p, jj, X, W, Y, coef, ws, dX, dW)
        torch.cuda.synchronize()
        print(json.dumps({"sample": jj, "masked_rows": int(m.sum()),
                          "device_error": list(bg.get_device_error(ws))}), flush=True)
    print(json.dumps({"workspace_bytes": ws.numel(),
                      "peak_mem_bytes": torch.cuda.max_memory_allocated()}), flush=True)


def grad_seed(wl, n_t, rep):
    """Draw seed of repeat `rep` at `n_t` (rep = -1: the golden gradient)."""
    return wl.seed + 1_000_003 if rep < 0 else wl.seed + 1 + 7919 * rep + 104729 * n_t


def grad_variance(bg, wl, nts, repeats, golden_nt, dev):
    """Sec. 4.3 on the synthetic head: the batch gradient dW of the on-policy
    BGPO objective computed `repeats` times with independent MC draws for each
    n_t; std = mean over parameters of the per-parameter std over the repeats,
    bias = mean over parameters of |mean over repeats - golden|, golden = the
    gradient with golden_nt samples."""
    import torch
    from synth import make_inputs
    inp = make_inputs(wl)
    X, W, Y = inp["X"].to(dev), inp["W"].to(dev), inp["Y"].to(dev)
    base = bg.problem_from(wl)
    A = torch.empty(wl.B, dtype=torch.float32, device=dev)
    if inp["A"] is not None:
        A.copy_(inp["A"].to(dev))
    else:
        bg.group_advantage(base, inp["rewards"].to(dev), A)
    dX = torch.zeros((wl.B, wl.R, wl.H), dtype=torch.float32, device=dev)
    dW = torch.zeros((wl.V, wl.H), dtype=torch.float32, device=dev)

    def gradient(n_t, seed):
        prob = bg.problem(wl.B, wl.P, wl.R, wl.H, wl.V, n_t, wl.G, wl.t_mode, seed)
        ws = bg.alloc_workspace(prob, dev)
        ell = torch.empty(wl.B, dtype=torch.float32, device=dev)
        coef = torch.empty_like(ell)
        dW.zero_()
        dX.zero_()
        for j in range(n_t):
            bg.sample_mask(prob, j, ws)
            bg.elbo_fwd(prob, j, X, W, Y, ws, ell)
            bg.bound_coeffs(prob, j, ell, ell, A, coef, None, ws)   # on-policy: d = 0
            bg.elbo_bwd_accumulate(prob, j, X, W, Y, coef, ws, dX, dW)
        code = bg.get_device_error(ws)[0]
        if code != 0:
            raise RuntimeError(f"device error {code}")
        return dW.double()

    golden = gradient(golden_nt, grad_seed(wl, golden_nt, -1)).clone()
    out = []
    for n_t in nts:
        s1 = torch.zeros_like(golden)
        s2 = torch.zeros_like(golden)
        for rep in range(repeats):
            g = gradient(n_t, grad_seed(wl, n_t, rep))
            s1 += g
            s2 += g * g
        mean = s1 / repeats
        var = (s2 / repeats - mean * mean).clamp_min(0.0)
        out.append({"n_t": n_t, "std": float(var.sqrt().mean()),
                    "bias": float((mean - golden).abs().mean())})
    return out


def run_grad_variance(args, wl):
    import torch
    import paper_2510_11683_gb300 as bg
    from paper_2510_11683_gb300 import build as B
    if not os.path.exists(B.LIB_PATH):
        B.build()
    dev = torch.device("cuda", 0)
    study = CONFIG_GRAD_VARIANCE
    t0 = time.perf_counter()
    wl = wl.with_(eps_std=0.0)   # on-policy: BGPO and VRPO gradients coincide (Sec. 3.2)
    res = grad_variance(bg, wl, study["n_t"], study["repeats"], study["golden_n_t"], dev)
    print(json.dumps({"experiment": "grad_std_bias_vs_n_t (Sec. 4.3)",
                      "workload": config_of(wl)["workload"], "repeats": study["repeats"],
                      "golden_n_t": study["golden_n_t"], "points": res,
                      "seconds": time.perf_counter() - t0}), flush=True)


CONFIG_GRAD_VARIANCE = {"n_t": (1, 2, 4, 8, 16, 32), "repeats": 8, "golden_n_t": 256}


def nt_sweep(bg, dev, pair=False):
    """Time and peak memory of one step vs n_t (8 x (256 + 512), LLaDA-8B head) for
    BGPO and for the ELBO-based objective it bounds (VRPO, Eq. 7), whose weights
    need every sample's l first: "vrpo_retain" keeps one workspace per sample
    (memory grows with n_t), "vrpo_recompute" runs each sample's forward twice.
    Every backward recomputes its logits. `pair`: BGPO and vrpo_recompute pair
    the dW GEMMs of samples 2k and 2k + 1 (vrpo_retain, one workspace per
    sample, cannot)."""
    import torch
    from synth import CONFIGS, SWEEP_NT, make_inputs
    base = CONFIGS["llada8b_sweep"]
    inp0 = make_inputs(base.with_(n_t=max(SWEEP_NT)))
    X, W, Y = inp0["X"].to(dev), inp0["W"].to(dev), inp0["Y"].to(dev)
    rewards = inp0["rewards"].to(dev)
    res = []
    for n_t in SWEEP_NT:
        wl = base.with_(n_t=n_t)
        prob = bg.problem_from(wl)
        A = torch.empty(wl.B, dtype=torch.float32, device=dev)
        bg.group_advantage(prob, rewards, A)
        rows = 0
        m = torch.empty((wl.B, wl.R), dtype=torch.uint8, device=dev)
        ws0 = bg.alloc_workspace(prob, dev)
        for j in range(n_t):
            bg.sample_mask(prob, j, ws0, None, m)
            rows += int(m.sum().item())
        del ws0
        point = {"n_t": n_t, "masked_rows": rows}
        for method in ("bgpo", "vrpo_retain", "vrpo_recompute"):
            torch.cuda.synchronize()
            torch.cuda.empty_cache()
            torch.cuda.reset_peak_memory_stats(dev)
            n_ws = n_t if method == "vrpo_retain" else 1
            pm = bg.problem_from(wl, pair_dw=pair and method != "vrpo_retain")
            wss = [bg.alloc_workspace(pm, dev) for _ in range(n_ws)]
            ell = torch.empty((n_t, wl.B), dtype=torch.float32, device=dev)
            coef, g = torch.empty_like(ell), torch.empty_like(ell)
            cv = torch.empty(wl.B, dtype=torch.float32, device=dev)
            tmp = torch.empty(wl.B, dtype=torch.float32, device=dev)
            dX = torch.zeros((wl.B, wl.R, wl.H), dtype=torch.float32, device=dev)
            dW = torch.zeros((wl.V, wl.H), dtype=torch.float32, device=dev)

            def run():
                if method == "bgpo":
                    ws = wss[0]
                    for j in range(n_t):
                        bg.sample_mask(pm, j, ws)
                        bg.elbo_fwd(pm, j, X, W, Y, ws, ell[j])
                        bg.bound_coeffs(pm, j, ell[j], ell[j], A, coef[j], g[j], ws)
                        bg.elbo_bwd_accumulate(pm, j, X, W, Y, coef[j], ws, dX, dW)
                    return
                for j in range(n_t):
                    ws = wss[j % n_ws]
                    bg.sample_mask(pm, j, ws)
                    bg.elbo_fwd(pm, j, X, W, Y, ws, ell[j])
                bg.vrpo_coeffs(pm, ell, ell, A, cv, None, wss[0])
                for j in range(n_t):
                    ws = wss[j % n_ws]
                    if method == "vrpo_recompute":
                        bg.sample_mask(pm, j, ws)
                        bg.elbo_fwd(pm, j, X, W, Y, ws, tmp)
                    bg.elbo_bwd_accumulate(pm, j, X, W, Y, cv, ws, dX, dW)
            run()
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            run()
            e1.record()
            torch.cuda.synchronize()
            ms = e0.elapsed_time(e1)
            code = bg.get_device_error(wss[0])[0]
            if code != 0:
                raise RuntimeError(f"n_t sweep {method}: device error {code}")
            point[method] = {"ms": ms, "tokens_per_s": rows / (ms / 1e3),
                             "peak_bytes": torch.cuda.max_memory_allocated(dev),
                             "dw_paired": bool(pm.flags & bg.FLAG_PAIR_DW)}
            del wss, dX, dW
        res.append(point)
    return res


if __name__ == "__main__":
    main()
