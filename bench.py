"""Throughput of one fused GRPO update step (scoring + loss + backward) on GB300.

A step is the whole path over one synthetic batch: group_advantages -> grpo_score_fwd ->
grpo_loss_bwd (logits, log-softmax at the sampled token, entropy, argmax, advantages, clipped
surrogate + KL loss, dL/dH and dL/dW). Default workload: 2 prompts x G=16 completions, T=16384,
lengths U{4096..16384}, d=5120, V=151936, bf16, per-token temperature U[0.5, 2].

Metric: scored tokens per second (fwd+bwd) and the algorithmic TFLOP/s (6 N d V per step) as a
fraction of the measured dense BF16 peak. Prints one JSON line (rank 0).

  python bench.py [--gpus N --steps K --warmup W --config NAME]
  python bench.py --impl reference ...   # the CPU float64 oracle on host cores, same metric
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

DEFAULT_CONFIG = "g16_t16k_d5120_v152k"
PEAKS_PATH = os.path.join(ROOT, "MEASURED_PEAKS.json")
PROFILES = os.path.join(ROOT, "profiles")
KERNEL_SRC = os.path.join(ROOT, "paper_2510_17158_gb300", "csrc", "gemm_tc.cu")
GEMM_KERNELS = ("fwd_gemm_tc", "bwd_dz_gemm_tc", "bwd_dh_gemm_tc", "bwd_dw_gemm_tc")



TILE_MODES = {0: "single CTA 128x256 (cta_group::1)",
              1: "CTA pair 256x256 (cta_group::2)",
              2: "CTA pair 256x512 (cta_group::2, two N=256 MMAs per k-step)"}

def tiles_desc(G):
    modes = [G.grpo_get_role_tile_mode(r) for r in range(4)]
    if len(set(modes)) == 1:
        return TILE_MODES[modes[0]]
    return "; ".join(f"{role}: {TILE_MODES[m]}" for role, m in zip(("fwd", "dz", "dH", "dW"), modes))


def peaks():
    try:
        p = json.load(open(PEAKS_PATH))
        return {"hbm_gbs": p["hbm_gbs"], "bf16": p["bf16_tflops"],
                "bf16_sustained": p["bf16_tflops_sustained"], "source": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16": 1900.0, "bf16_sustained": 1700.0, "source": "fallback"}


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def dist_init(ws, backend):
    if ws > 1:
        import torch.distributed as dist
        if not dist.is_initialized():
            dist.init_process_group(backend=backend)


def dist_max(x: float, ws: int, device) -> float:
    if ws == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def dist_sum(x: float, ws: int, device) -> float:
    if ws == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def barrier(ws):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


def dp_exchange(bwd_out: dict, ws: int):
    """The data-parallel step's one exchange: every rank scored its own whole groups with the
    global normaliser, so the summed loss and dW are the single-process ones; dH rows stay with
    the rank that owns them. Issued on the current stream, inside the timed step."""
    if ws > 1:
        import torch.distributed as dist
        dist.all_reduce(bwd_out["dW"], op=dist.ReduceOp.SUM)
        dist.all_reduce(bwd_out["loss"], op=dist.ReduceOp.SUM)
    return bwd_out


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples every 200 ms while the timed region runs."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        self.out = ""
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        rows = []
        for line in (self.out or "").strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                rows.append((float(f[1]), float(f[2]), float(f[3]), f[5], f[6], f[7], f[8]))
            except ValueError:
                continue
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        loaded = [r for r in rows if r[2] > 200.0] or rows
        reasons = set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for r in loaded:
            for n, v in zip(names, r[3:]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(r[0] for r in loaded),
                "sm_max_mhz": max(r[1] for r in rows), "samples": len(loaded),
                "power_w_max": max(r[2] for r in rows), "reasons": sorted(reasons)}


def kernel_source_sha() -> str:
    """Hash of the GEMM kernel's code with comments and blank lines removed (a comment edit does
    not invalidate a committed traffic measurement; any code change does)."""
    txt = open(KERNEL_SRC).read()
    txt = re.sub(r"//[^\n]*", "", txt)
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    txt = "\n".join(line.strip() for line in txt.splitlines() if line.strip())
    return hashlib.sha256(txt.encode()).hexdigest()[:16]


def ncu_traffic(kernel: str, workload: str, tile_mode: int):
    """DRAM bytes per launch from a committed ncu summary of this kernel, if it was taken on the
    current kernel source in the tile mode the kernel runs in now (profiles/<kernel>__<workload>.md
    with 'source_sha', 'tile_mode' and 'dram_bytes_per_launch_full' lines; a summary without a
    'tile_mode' line was taken with single-CTA tiles)."""
    path = os.path.join(PROFILES, f"{kernel}__{workload}.md")
    if not os.path.exists(path):
        return None
    txt = open(path).read()
    sha = re.search(r"source_sha:\s*([0-9a-f]+)", txt)
    val = re.search(r"dram_bytes_per_launch_full:\s*([0-9.eE+]+)", txt)
    mode = re.search(r"tile_mode:\s*(-?[0-9]+)", txt)
    if not sha or not val or sha.group(1) != kernel_source_sha():
        return None
    if (int(mode.group(1)) if mode else 0) != tile_mode:
        return None
    return float(val.group(1))


def apply_scale(w, spec: str):
    if not spec:
        return w
    kw = {}
    for item in spec.split(","):
        k, v = item.split("=")
        kw[k] = tuple(int(x) for x in v.split("/")) if k == "group_sizes" else int(v)
    return w.scaled(name=w.name + "_scaled", **kw)


# ---------------------------------------------------------------------------------------------
def run_reference(args, ws_size, rank):
    """The CPU float64 oracle, as it stands, timed on this host's cores on a bounded sample of the
    workload (a slice of scored tokens of the first completion, full d and V)."""
    if rank != 0:
        return
    from paper_2510_17158_gb300.synthetic import WORKLOADS
    w = apply_scale(WORKLOADS[args.config], args.scale)
    line = cpu_baseline(w, args.ref_tokens, steps=args.steps, warmup=args.warmup)
    value = line["value"]
    out = {"metric": "scored tokens/sec (fwd+bwd)", "value": value, "unit": "tokens/s",
           "n_gpus": ws_size, "steps": args.steps, "warmup": args.warmup,
           "ms_per_step": line["ms_per_step"], "higher_is_better": True, "scaling": "weak",
           "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
           "config": {"workload": w.name, "prompts": w.prompts, "G": list(w.group_sizes), "T": w.T,
                      "d": w.d, "V": w.V},
           "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": line["cores"],
                            "kind": "oracle", "sample": line["sample"]},
           "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def blas_threads() -> int:
    """Threads the oracle's numpy BLAS runs with (torch.distributed.run sets OMP_NUM_THREADS=1
    in every rank unless the caller set it)."""
    try:
        from threadpoolctl import threadpool_info
        n = [p["num_threads"] for p in threadpool_info() if p.get("user_api") == "blas"]
        if n:
            return int(max(n))
    except Exception:
        pass
    for k in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS"):
        if os.environ.get(k, "").isdigit():
            return int(os.environ[k])
    return os.cpu_count()


def cpu_baseline(w, n_tokens, steps=1, warmup=0):
    """Times oracle.grpo_step (fwd + loss + dH + full dW) on the first `n_tokens` positions of
    one completion of workload `w` (inputs drawn with the workload's laws), float64 on host cores."""
    import oracle
    rng = np.random.default_rng(w.seed)
    d, V = w.d, w.V
    H = rng.standard_normal((1, n_tokens, d)).astype(np.float32)
    H /= np.sqrt((H.astype(np.float64) ** 2).mean(-1, keepdims=True)).astype(np.float32)
    if w.temperature:
        H /= rng.uniform(*w.temperature, size=(1, n_tokens, 1)).astype(np.float32)
    tdt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    H = torch.from_numpy(H).to(tdt).double().numpy()
    W = torch.from_numpy((rng.standard_normal((V, d), dtype=np.float32) * 0.02)).to(tdt).double().numpy()
    tokens = rng.integers(0, V, size=(1, n_tokens)).astype(np.int32)
    mask = np.ones((1, n_tokens), np.uint8)
    old = rng.normal(-8, 1, size=(1, n_tokens))
    ref = old + rng.normal(0, 0.1, size=(1, n_tokens))
    rewards = np.array([1.0], np.float32)
    go = np.array([0, 1], np.int32)
    times = []
    for it in range(warmup + steps):
        t0 = time.perf_counter()
        oracle.grpo_step(H, W, tokens, mask, rewards, go, old, ref, w.eps, w.eps, w.beta)
        if it >= warmup:
            times.append(time.perf_counter() - t0)
    per = sum(times) / len(times)
    nthr = blas_threads()
    return {"value": n_tokens / per, "ms_per_step": per * 1e3, "cores": nthr,
            "sample": f"{n_tokens} scored tokens of one completion, full d={d}, V={V} "
                      f"(fwd + loss + dH + full dW), float64 numpy on {nthr} host "
                      f"threads; mean of {len(times)} run(s)"}


def run_e2e(step, dev_args, stream, device, e2e_steps, ws_n):
    """Times `e2e_steps` steps whose inputs come from pinned host memory (double-buffered copies
    on a second stream) and whose loss is read back; returns (seconds, host->device bytes/step)."""
    names = ("H", "W", "tokens", "mask", "rewards", "go", "old", "ref")
    host = {k: v.cpu().pin_memory() for k, v in zip(names, dev_args)}
    h2d = sum(v.numel() * v.element_size() for v in host.values())
    sets = [dev_args, tuple(torch.empty_like(v) for v in dev_args)]
    copy_stream = torch.cuda.Stream(device)
    copied = [torch.cuda.Event(), torch.cuda.Event()]
    used = [torch.cuda.Event(), torch.cuda.Event()]
    loss_host = torch.empty(e2e_steps, dtype=torch.float32).pin_memory()

    def upload(j):
        with torch.cuda.stream(copy_stream):
            if j >= 2:
                copy_stream.wait_event(used[j % 2])     # step j-2 is done with this set
            for k, dst in zip(names, sets[j % 2]):
                dst.copy_(host[k], non_blocking=True)
            copied[j % 2].record(copy_stream)

    torch.cuda.synchronize()
    barrier(ws_n)
    t0 = time.perf_counter()
    upload(0)
    for j in range(e2e_steps):
        if j + 1 < e2e_steps:
            upload(j + 1)
        stream.wait_event(copied[j % 2])
        r = step(*sets[j % 2])
        used[j % 2].record(stream)
        loss_host[j:j + 1].copy_(r["loss"], non_blocking=True)
    torch.cuda.synchronize()
    e2e_s = time.perf_counter() - t0
    barrier(ws_n)
    e2e_s = dist_max(e2e_s, ws_n, device)
    if not bool(torch.isfinite(loss_host).all()):
        raise RuntimeError("non-finite loss in the end-to-end steps")
    return e2e_s, h2d


# ---------------------------------------------------------------------------------------------
def run_gpu(args):
    ws_n, rank, local = dist_env()
    device = torch.device(f"cuda:{local}")
    torch.cuda.set_device(device)
    dist_init(ws_n, "nccl")
    from paper_2510_17158_gb300 import grpo as G
    from paper_2510_17158_gb300.synthetic import WORKLOADS, lm_head_flops, make_batch_torch
    G.grpo_set_tile_mode(args.tile_mode)
    if args.role_tile_modes:
        role_modes = [int(x) for x in args.role_tile_modes.split(",")]
        if len(role_modes) != 4:
            raise SystemExit("--role-tile-modes wants four comma-separated modes (fwd,dz,dH,dW)")
        for role, m in enumerate(role_modes):
            G.grpo_set_role_tile_mode(role, m)
    win = None
    if args.gemm_window:
        win = [int(x) for x in args.gemm_window.split(",")]
        G.grpo_set_gemm_window(win[0], win[1])
    w = apply_scale(WORKLOADS[args.config], args.scale)
    w = w.scaled(seed=w.seed + 1000 * rank)        # each rank scores its own groups
    if args.beta is not None:
        w = w.scaled(beta=args.beta)
    t_gen = time.time()
    b = make_batch_torch(w, device=str(device))
    S, T, d, V = w.S, w.T, w.d, w.V
    N_v = int(b.mask.sum().item())
    ws = G.Workspace.for_problem(S, T, d, V, b.H.dtype, vocab_chunk=args.vocab_chunk,
                                 device=device, kl=args.path == "grpo-exact-kl")
    stream = torch.cuda.current_stream(device)
    # old / ref log-probs: the policy's own log-prob (a scoring pass) plus the workload's noise
    f0 = G.grpo_score_fwd(b.H, b.W, b.tokens, b.mask, ws)
    old = (f0["logp"] + b.noise_old).contiguous()
    ref = (f0["logp"] + b.noise_ref).contiguous()
    fwd_out = {k: torch.empty_like(v) for k, v in f0.items()}
    if args.path == "grpo-exact-kl":
        from paper_2510_17158_gb300.synthetic import reference_model_inputs
        H_ref, W_ref = reference_model_inputs(b)
        fwd_out["lse_ref"] = torch.empty_like(f0["lse"])
        fwd_out["kl"] = torch.empty_like(f0["lse"])
    bwd_out = {"loss": torch.empty(1, device=device), "dH": torch.empty_like(b.H),
               "dW": torch.empty((V, d), dtype=torch.float32, device=device)}
    adv = torch.empty(S, device=device)
    # loss normaliser over all ranks (Eq. 1's expectation over every rank's sequences, or every
    # scored token for the distillation loss); 0 = this batch's own count
    norm = 0.0
    if ws_n > 1:
        from paper_2510_17158_gb300 import dp
        norm = dp.global_norm("token_mean" if args.path == "sft" else "seq_mean", S, N_v,
                              lambda x: dist_sum(x, ws_n, device))
        if args.graph:
            raise SystemExit("--graph with more than one rank: the dW all-reduce is not captured")
    torch.cuda.synchronize()
    gen_s = time.time() - t_gen

    def step(H, W, tok, mask, rewards, go, old_, ref_):
        if args.path == "grpo-exact-kl":   # Eq. 1's KL over the whole vocabulary
            G.group_advantages(rewards, go, ws, adv_out=adv)
            f = G.grpo_score_fwd_kl(H, W, H_ref, W_ref, tok, mask, ws, out=fwd_out)
            o = G.grpo_loss_bwd_kl(H, W, H_ref, W_ref, tok, mask, f, old_, adv, ws,
                                   eps_low=w.eps, eps_high=w.eps, beta=w.beta, norm=norm,
                                   out=bwd_out)
        elif args.path == "sft":     # distillation step (Sec. 6.2): no advantages, no ratio
            f = G.grpo_score_fwd(H, W, tok, mask, ws, out=fwd_out)
            o = G.grpo_sft_loss_bwd(H, W, tok, mask, f["logp"], f["lse"], f["valid_count"],
                                    ws, norm=norm, out=bwd_out)
        else:
            G.group_advantages(rewards, go, ws, adv_out=adv)
            f = G.grpo_score_fwd(H, W, tok, mask, ws, out=fwd_out)
            if w.beta == 0.0:      # no KL term: the reference log-probs are not read
                ref_ = None
            o = G.grpo_loss_bwd(H, W, tok, mask, f["logp"], f["lse"], old_, ref_, adv,
                                f["valid_count"], ws, eps_low=w.eps, eps_high=w.eps,
                                beta=w.beta, norm=norm, out=bwd_out)
        return dp_exchange(o, ws_n)

    dev_args = (b.H, b.W, b.tokens, b.mask, b.rewards, b.group_offsets, old, ref)
    for _ in range(args.warmup):
        step(*dev_args)
    graph = None
    launches_per_graph = 0
    if args.graph:      # the whole step as one CUDA graph (all launches replayed at once)
        torch.cuda.synchronize()
        G.grpo_timing_reset()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            step(*dev_args)
        launches_per_graph = sum(n for n, _ in G.timing_table().values())
        graph.replay()
    torch.cuda.synchronize()
    st, where = G.grpo_last_device_error(ws)
    if st != 0:
        raise RuntimeError(f"device status {st} at {where} during warm-up")

    # ---- device-resident timed region --------------------------------------------------------
    G.grpo_timing_reset()
    G.grpo_timing_enable(True)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(device.index if device.index is not None else 0) as clk:
        barrier(ws_n)
        torch.cuda.synchronize()
        ev0.record(stream)
        for _ in range(args.steps):
            if graph is not None:
                graph.replay()
            else:
                step(*dev_args)
        ev1.record(stream)
        torch.cuda.synchronize()
        barrier(ws_n)
    G.grpo_timing_enable(False)
    ms = ev0.elapsed_time(ev1)
    ms_max = dist_max(ms, ws_n, device)
    table = G.timing_table()
    launches = sum(n for n, _ in table.values())
    if graph is not None:    # replays record no per-kernel events; launches come from the capture
        launches = launches_per_graph * args.steps
    st, where = G.grpo_last_device_error(ws)
    if st != 0:
        raise RuntimeError(f"device status {st} at {where} in the timed region")

    # ---- end to end through the public API with host buffers --------------------------------
    # Every step's inputs are copied from pinned host memory and its loss read back inside the
    # timed region. Inputs are double-buffered: step j+1's copies run on a second stream while
    # step j computes (GB300's C2C link moves the 6.9 GB in a few percent of a step).
    # --e2e-steps 0 skips this part (profiling captures: no second copy of the inputs).
    e2e_steps = args.e2e_steps
    e2e_s = h2d = None
    if e2e_steps > 0:
        e2e_s, h2d = run_e2e(step, dev_args, stream, device, e2e_steps, ws_n)

    total_tokens = dist_sum(float(N_v), ws_n, device)
    value = total_tokens * args.steps / (ms_max / 1e3)
    e2e_value = total_tokens * e2e_steps / e2e_s if e2e_steps > 0 else None
    pk = peaks()
    step_ms = ms_max / args.steps
    # algorithmic flop per step: 6 N d V (fwd, dH, dW); the exact-KL path adds the reference
    # model's forward product (8 N d V). Recomputed products count as overhead, not work.
    alg_flop = lm_head_flops(N_v, d, V) * (8.0 / 6.0 if args.path == "grpo-exact-kl" else 1.0)
    alg_tflops = alg_flop / (step_ms / 1e3) / 1e12

    # ---- roofline of the dominant kernel -------------------------------------------------------
    per_kernel = {k: {"launches": n, "ms_total": round(t, 3), "ms_per_launch": round(t / n, 4),
                      "share": round(t / ms, 4)} for k, (n, t) in table.items()}
    if not table:            # graph replays: no per-kernel timing
        table = {"graph_replay": (args.steps, ms)}
    dom = max(table, key=lambda k: table[k][1])
    n_dom, t_dom = table[dom]
    kl2 = 2.0 if args.path == "grpo-exact-kl" else 1.0
    # algorithmic flop of each GEMM per step, summed over its launches (one per vocabulary chunk
    # for dz, dH and dW; the last chunk may be narrower); rates = timed-region flop / kernel time
    flops_per_step = {
        "fwd_gemm_tc": 2.0 * kl2 * N_v * d * V, "bwd_dz_gemm_tc": 2.0 * kl2 * N_v * d * V,
        "bwd_dh_gemm_tc": 2.0 * N_v * d * V, "bwd_dw_gemm_tc": 2.0 * N_v * d * V}
    if dom in flops_per_step:
        achieved = flops_per_step[dom] * args.steps / (t_dom / 1e3) / 1e12
        roof = {"kernel": dom, "bound": "tensor", "achieved": round(achieved, 1),
                "peak": pk["bf16_sustained"], "unit": "TFLOP/s",
                "frac": round(achieved / pk["bf16_sustained"], 4),
                "peak_source": f"{pk['source']} bf16 sustained (kernel timed inside a long step)",
                # committed ncu summaries cover the GRPO path's own GEMMs
                "traffic": (ncu_traffic(dom, w.name, G.grpo_get_role_tile_mode(GEMM_KERNELS.index(dom)))
                            if args.path == "grpo" and not args.vocab_chunk else None)}
    else:
        roof = {"kernel": dom, "bound": "hbm", "achieved": None, "peak": pk["hbm_gbs"],
                "unit": "GB/s", "frac": None, "traffic": None}
    gemm_tf = {}
    for k in GEMM_KERNELS:
        if k in table:
            n, t = table[k]
            gemm_tf[k] = round(flops_per_step[k] * args.steps / (t / 1e3) / 1e12, 1)

    out = {
        "metric": "scored tokens/sec (fwd+bwd)" + {"sft": " [SFT distillation step]",
                                                    "grpo-exact-kl": " [GRPO, exact KL]"}.get(
                                                        args.path, ""),
        "value": round(value, 1), "unit": "tokens/s", "n_gpus": ws_n, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(step_ms, 3), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": w.name, "prompts": w.prompts, "G": list(w.group_sizes), "T": T,
                   "d": d, "V": V, "eps": w.eps, "beta": w.beta, "scored_tokens_per_rank": N_v,
                   "vocab_chunk": args.vocab_chunk or "whole vocabulary",
                   "tiles": tiles_desc(G),
                   "gemm_window": ("library default (dH, dW: a barrier every 256 k-blocks)"
                                   if win is None else "off" if win[0] == 0 else
                                   f"{win[0]} k-blocks, lag {win[1]} checkpoints" if win[0] > 0
                                   else f"every {-win[0]} work unit(s), lag {win[1]}"),
                   "l2": "inputs larger than L2 (H %.2f GB, W %.2f GB resident in HBM)" % (
                       b.H.numel() * 2 / 1e9, b.W.numel() * 2 / 1e9),
                   "parallelism": (f"dp{ws_n} (whole groups per GPU, global loss normaliser; dW "
                                   "and loss all-reduced over NCCL every step)" if ws_n > 1 else
                                   "dp1"),
                   "cuda_graph": bool(args.graph)},
        "tflops_alg": round(alg_tflops, 1),
        "frac_of_bf16_peak": round(alg_tflops / pk["bf16"], 4),
        "frac_of_bf16_sustained": round(alg_tflops / pk["bf16_sustained"], 4),
        "gemm_tflops_alg": gemm_tf,
        "roofline": roof,
        "kernels": per_kernel,
        "gpu_launches": launches,
        "e2e": None if e2e_value is None else {
            "value": round(e2e_value, 1), "unit": "tokens/s", "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": 4, "steps": e2e_steps,
            "copies": "pinned host -> device every step; step j+1's inputs copied on a "
                      "second stream while step j computes"},
        "clocks": clk.summary(),
        "setup_s": round(gen_s, 1),
    }
    if rank == 0 and ws_n == 1 and not args.no_cpu_baseline:
        cb = cpu_baseline(w, args.cpu_tokens)
        out["cpu_baseline"] = {"value": round(cb["value"], 2), "unit": "tokens/s",
                               "cores": cb["cores"], "kind": "oracle", "sample": cb["sample"]}
    if rank == 0:
        print(json.dumps(out), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1,
                    help="GPUs (one process each); without WORLD_SIZE in the environment, N > 1 "
                         "re-launches this command under torch.distributed.run")
    ap.add_argument("--master-port", type=int, default=29533)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--config", default=DEFAULT_CONFIG)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--vocab-chunk", type=int, default=0,
                    help="vocabulary columns of dz kept at once (0 = whole vocabulary)")
    ap.add_argument("--beta", type=float, default=None,
                    help="KL coefficient (default: the workload's); 0 = no KL term, reference "
                         "log-probs not read")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--cpu-tokens", type=int, default=32)
    ap.add_argument("--ref-tokens", type=int, default=16)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--path", default="grpo", choices=["grpo", "sft", "grpo-exact-kl"],
                    help="grpo: the GRPO update (default); sft: the distillation loss step; "
                         "grpo-exact-kl: GRPO with the full-vocabulary KL to a reference model")
    ap.add_argument("--tile-mode", type=int, default=-1, choices=[-1, 0, 1, 2],
                    help="tensor-core tiles of every GEMM: -1 = the library's per-GEMM default "
                         "(fwd 0, dz 0, dH 2, dW 2); "
                         + "; ".join(f"{k} = {v}" for k, v in TILE_MODES.items()))
    ap.add_argument("--role-tile-modes", default="",
                    help="per-GEMM tile modes fwd,dz,dH,dW, applied after --tile-mode "
                         "(-1 = that GEMM's default)")
    ap.add_argument("--gemm-window", default="",
                    help="progress window of the dH and dW GEMMs CHECK,LAG: producers stay within "
                         "LAG checkpoints of the launch's average; checkpoints every CHECK "
                         "k-blocks, or at every -CHECK-th work unit for CHECK < 0 (write "
                         "--gemm-window=-1,1); '0,0' = off; default: the library's (256,1)")
    ap.add_argument("--graph", action="store_true",
                    help="capture one step in a CUDA graph and time its replays (per-kernel "
                         "timing and launch counts then come from the capture, not the replays)")
    ap.add_argument("--scale", default="",
                    help="override workload fields, e.g. 'prompts=1,group_sizes=2,T=2048' "
                         "(for profiling captures on a smaller case)")
    args = ap.parse_args()
    if args.impl == "ours":
        args.warmup = max(3, args.warmup)      # timing rule: at least 3 warm-up steps
    if args.gpus > 1 and "WORLD_SIZE" not in os.environ:
        # one process per GPU: re-launch this command under torch.distributed.run
        cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1",
               f"--nproc-per-node={args.gpus}", "--master-addr=127.0.0.1",
               f"--master-port={args.master_port}", os.path.abspath(__file__)] + sys.argv[1:]
        raise SystemExit(subprocess.call(cmd))
    ws_n, rank, _ = dist_env()
    if ws_n != args.gpus:
        raise SystemExit(f"--gpus {args.gpus} but WORLD_SIZE={ws_n}")
    if args.impl == "reference":
        run_reference(args, ws_n, rank)
        return
    run_gpu(args)


if __name__ == "__main__":
    main()
