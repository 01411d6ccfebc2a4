"""Benchmark of the REFLEX per-forward MoE hot path on GB300.

Default workload (one step = one whole denoising forward): a stack of 16
LLaDA-MoE-shaped MoE layers (d = 2048, E = 64 SwiGLU experts with inter =
1024, K in [2, 12], bf16 storage, fp32 accumulation) over a batch of 32 x
1024 tokens (512 prompt + 512 generated, blocks of 32).  The per-token counts
are allocated once per forward (Eq. 3 realised by Eq. 5, Eq. 6-9 and the
clip) and shared by every layer (Sec. 3.3); each layer runs the
variable-count layer of Eq. 2 (router scores, variable-count TopK, pair
dispatch, grouped SwiGLU expert GEMMs on tcgen05, weighted combine) with the
residual h <- bf16(h + MoE(h)).  Inputs are synthetic and seeded on the host
(the oracle can check the exact timed inputs).

Prints ONE JSON line (rank 0).  `value` = tokens/s of whole forwards over all
ranks; `expert_tflops` = 6 d inter sum(k) x layers / forward time (Eq. 10);
the same kernels at fixed top-K_base run beside it; `roofline` is for the
dominant kernel, the CTA-pair gate/up (SwiGLU) GEMM; `e2e` times the same
forward from pinned host buffers through the public API with the copies
inside the timed region; `cpu_baseline` times the oracle on the host cores.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reflex|reference]
                  [--config NAME] [--no-cpu-baseline] [--sweep [--sweep-tokens
                  T1,T2..] [--sweep-skews S1,S2..]] [--ablation] [--trajectory]
--config llada_moe | llada2_mini | llada_moe_b32 | tiny_fp32: one layer, one
reflex_step call (counts + layer) per step.
--sweep: LLaDA2.0-mini layer shapes, 256 .. 65536 tokens x count skew
0 .. 1 (0 = uniform K_base, 1 = 70% K_min / 30% K_max), forward only; the
token counts and skews can be listed instead.
Under torchrun each rank runs its own batch on its own GPU (weak scaling, no
data-path collective; a barrier and a max-reduce of the times only).
"""
from __future__ import annotations

import argparse
import json
import os
import re
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2608_01784_gb300 import replicas as R  # noqa: E402
from paper_2608_01784_gb300 import workloads as W  # noqa: E402

METRIC = ("MoE-layer tokens/s and expert TFLOP/s (frac of roofline) REFLEX vs "
          "fixed top-K")

# DRAM bytes (read + write) per launch of the dominant kernel, from one ncu
# capture of that kernel on the workload, with the SHA-256 prefix of the
# kernel source it was taken on; once the source differs the line reports
# null (the counters no longer describe the kernel that ran).
NCU_TRAFFIC = {
    "llada_moe": (561207296, "f1ace3cfdb36717b"),
    "llada2_mini": (1280278784, "f1ace3cfdb36717b"),
    "llada_moe_stack16": (1634616064, "f1ace3cfdb36717b"),
}
KERNEL_SOURCE = os.path.join(ROOT, "paper_2608_01784_gb300", "csrc", "experts_tc.cu")


def code_of(text: str) -> str:
    """C++ source without comments and with whitespace runs collapsed: what
    the compiler sees of it (string literals hold no comment markers here)."""
    text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
    text = re.sub(r"//[^\n]*", " ", text)
    return " ".join(text.split())


def kernel_source_sha16() -> str:
    """SHA-256 prefix of the GEMM source's code (comments and layout
    ignored), the key the DRAM-traffic captures are kept under."""
    import hashlib
    with open(KERNEL_SOURCE, encoding="utf-8") as f:
        return hashlib.sha256(code_of(f.read()).encode()).hexdigest()[:16]


def ncu_traffic(workload: str):
    nbytes, sha = NCU_TRAFFIC.get(workload, (None, None))
    if nbytes is None or sha != kernel_source_sha16():
        return None
    return nbytes


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="reflex", choices=["reflex", "reference"])
    ap.add_argument("--config", default="llada_moe_stack16",
                    choices=sorted(W.CONFIGS) + ["llada_moe_stack16"])
    ap.add_argument("--sweep", action="store_true",
                    help="token-count x count-skew sweep on the LLaDA2.0-mini "
                         "layer (one JSON line per point)")
    ap.add_argument("--sweep-tokens", default=None,
                    help="comma-separated token counts of --sweep (default 256 .. "
                         "65536, doubling)")
    ap.add_argument("--sweep-skews", default=None,
                    help="comma-separated count skews of --sweep (default 0, 0.25, "
                         "0.5, 0.75, 1)")
    ap.add_argument("--trajectory", action="store_true",
                    help="whole denoising trajectories: NFE and pairs per sample")
    ap.add_argument("--ablation", action="store_true",
                    help="REFLEX and its App. C allocation ablations on one layer")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--gather-in-gemm", action="store_true",
                    help="fused dispatch: the CTA-pair gate/up GEMM gathers its "
                         "rows (REFLEX_FLAG_GATHER_IN_GEMM; slower, off by default)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="target seconds of oracle work for cpu_baseline")
    return ap.parse_args()


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return dict(hbm=d["hbm_gbs"], bf16=d["bf16_tflops"],
                    bf16_sustained=d.get("bf16_tflops_sustained"),
                    source="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sustained=1700.0, source="fallback")


# ---------------------------------------------------------------------------
# clocks sampled during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,"
              "clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            time.sleep(1.0)   # nvidia-smi takes a moment before its first sample
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return dict(sm_mhz=None, sm_max_mhz=None, reasons=[], samples=0)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out = ""
        sm, mx, pw, reasons = [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown",
                 "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
                pw.append(float(f[3]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        # under load: samples drawing at least half of the largest power seen
        top = max(pw) if pw else 0.0
        loaded = [c for c, w in zip(sm, pw) if w >= 0.5 * top]
        return dict(sm_mhz=statistics.median(loaded) if loaded else None,
                    sm_max_mhz=max(mx) if mx else None,
                    reasons=sorted(reasons), samples=len(sm),
                    samples_under_load=len(loaded),
                    power_w_max=top if pw else None)


# ---------------------------------------------------------------------------
# CPU oracle leg (cpu_baseline and --impl reference)
# ---------------------------------------------------------------------------
def oracle_step(cfg, layer, state, tokens):
    """The oracle's whole path for the listed tokens: allocation (whole batch;
    the count rule couples the tokens of an active block), router scores,
    TopK / alpha, pair order, Eq. 2."""
    import oracle
    k = oracle.allocate(state["conf1"], state["conf2"], state["hist_len"],
                        state["masked"], state["block_id"], state["seq_offsets"],
                        state["active_block"], **cfg.alloc_params())
    h = layer["hidden"][tokens]
    z = oracle.router_logits(h, layer["w_router"])
    ks = k[tokens]
    ids, alpha = oracle.select(z, ks, cfg.k_max)
    oracle.permutation(ids, ks, cfg.E)
    sub = np.arange(len(tokens), dtype=np.int32)
    oracle.moe_tokens(h, layer["w_gate_up"], layer["w_down"], ids, alpha, ks, sub,
                      shared_gate_up=layer.get("shared_gate_up"),
                      shared_down=layer.get("shared_down"))
    return int(ks.sum())


def oracle_rate(cfg, layer, state, target_s, seed=0, threads=None):
    """tokens/s of the oracle on a seeded token sample sized to ~target_s;
    threads = None keeps the OpenMP default (all cores)."""
    import oracle
    oracle.build()
    all_cores = oracle.num_threads()
    if threads is not None:
        oracle.set_num_threads(threads)
    try:
        used = oracle.num_threads()
        T = layer["hidden"].shape[0]
        rng = np.random.default_rng(seed)
        n = min(T, max(2, 2 * used))
        t0 = time.perf_counter()
        oracle_step(cfg, layer, state, np.sort(rng.choice(T, n, replace=False)).astype(np.int32))
        dt = time.perf_counter() - t0
        n2 = int(min(T, max(n, n * target_s / max(dt, 1e-6))))
        toks = np.sort(rng.choice(T, n2, replace=False)).astype(np.int32)
        t0 = time.perf_counter()
        oracle_step(cfg, layer, state, toks)
        dt = time.perf_counter() - t0
    finally:
        oracle.set_num_threads(all_cores)
    return n2 / dt, n2, dt, used


def layer_config(cfg, world: int) -> dict:
    return dict(workload=cfg.name, description=cfg.description, tokens_per_step=cfg.T,
                parallelism=f"replicas{world}",
                l2="no flush: expert weights > 129 MB L2 stream from HBM every step")


def run_reference(args, cfg, rank, world):
    import torch  # noqa: F401  (keeps the launch environment identical)
    if rank != 0:
        return
    layer = W.make_layer(cfg, args.seed)
    state = W.make_state(cfg, args.seed)
    import oracle
    oracle.build()
    T = cfg.T
    rng = np.random.default_rng(args.seed)
    # per step: a seeded token sample sized so that W + K steps stay within a
    # few minutes
    per_step_s = max(0.5, min(5.0, 150.0 / max(1, args.steps + args.warmup)))
    n = min(T, 8)
    t0 = time.perf_counter()
    oracle_step(cfg, layer, state, np.arange(n, dtype=np.int32))
    dt = time.perf_counter() - t0
    n = int(min(T, max(1, n * per_step_s / max(dt, 1e-6))))
    for _ in range(args.warmup):
        oracle_step(cfg, layer, state, np.sort(rng.choice(T, n, replace=False)).astype(np.int32))
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle_step(cfg, layer, state, np.sort(rng.choice(T, n, replace=False)).astype(np.int32))
    dt = time.perf_counter() - t0
    value = n * args.steps / dt
    line = dict(metric=METRIC, value=value, unit="tokens/s",
                impl="reference", n_gpus=args.gpus, steps=args.steps,
                warmup=args.warmup, ms_per_step=1e3 * dt / args.steps,
                higher_is_better=True, scaling="weak", vs_baseline=None,
                dtype="f64", data="synthetic",
                config=layer_config(cfg, world),
                cpu_baseline=dict(value=value, unit="tokens/s", kind="oracle",
                                  cores=oracle.num_threads(),
                                  sample=f"{n} seeded tokens of the {T}-token "
                                         f"batch per step (allocation on the "
                                         f"whole batch)"),
                e2e=dict(value=value, unit="tokens/s", h2d_bytes_per_step=0,
                         d2h_bytes_per_step=0))
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# GPU leg
# ---------------------------------------------------------------------------
def run_gpu(args, cfg, rank, world, local_rank):
    import torch
    from paper_2608_01784_gb300 import _binding as B
    from paper_2608_01784_gb300 import api, build

    build.build()
    B.load()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    seed = R.rank_seed(args.seed, rank)
    layer = W.make_layer(cfg, seed)
    state = W.make_state(cfg, seed)
    T, d, E, I, S, km = cfg.T, cfg.d, cfg.E, cfg.inter, cfg.shared_inter, cfg.k_max
    dl = api.layer_to_device(layer, cfg.dtype, dev)
    ds = api.state_to_device(state, dev)
    moe = api.MoELayer(dl, dtype=cfg.dtype, d=d, E=E, inter=I, shared_inter=S,
                       k_max=km, max_tokens=T, device=dev)
    stream = torch.cuda.current_stream(dev)
    p_reflex = B.make_params(**cfg.alloc_params())
    p_fixed = B.make_params(**cfg.alloc_params(delta_role=0, delta_cur=0))
    k_buf = torch.empty(T, dtype=torch.int32, device=dev)
    k_sum = torch.zeros(1, dtype=torch.int64, device=dev)
    st = torch.zeros(1, dtype=torch.int32, device=dev)
    out = torch.empty((T, d), dtype=moe.tdtype, device=dev)
    F = B.REFLEX_FLAG_RENORM_TOPK | (B.REFLEX_FLAG_GATHER_IN_GEMM if args.gather_in_gemm else 0)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]

    # every call takes the current stream, so the steps can be captured into
    # CUDA graphs (the library never synchronises with the host)
    def step(params, hidden=None):
        moe.step(ds, params, dl["hidden"] if hidden is None else hidden, out=out,
                 k_out=k_buf, k_sum=k_sum, status=st, flags=F)

    def staged_step(params, up_events):
        # the same work as step(), split so that events bracket the gate/up GEMM
        h = dl["hidden"]
        moe.step(ds, params, h, out=out, k_out=k_buf, k_sum=k_sum, status=st,
                 flags=F | B.REFLEX_STAGE_ROUTE | B.REFLEX_STAGE_DISPATCH)
        up_events[0].record()
        moe.forward(h, k_buf, out, F | B.REFLEX_STAGE_EXPERT_UP)
        up_events[1].record()
        moe.forward(h, k_buf, out, F | B.REFLEX_STAGE_EXPERT_DOWN | B.REFLEX_STAGE_COMBINE)

    def graph_of(fn):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, capture_error_mode="relaxed"):
            fn()
        return g

    def barrier():
        R.barrier(world, dev)

    def timed(graph, replays, warmup):
        for _ in range(warmup):
            graph.replay()
        barrier()
        start, stop = (torch.cuda.Event(enable_timing=True) for _ in range(2))
        start.record(stream)
        for _ in range(replays):
            graph.replay()
        stop.record(stream)
        barrier()
        return start.elapsed_time(stop)

    def max_over_ranks(x: float) -> float:
        return R.max_over_ranks(x, world, dev)

    # clocks sampled from the first launch to the end of the end-to-end leg
    clk = ClockSampler(local_rank)
    clk.start()
    # correctness gate before timing: counts and routing status clean
    step(p_reflex)
    torch.cuda.synchronize(dev)
    assert B.reflex_read_status(st) == B.REFLEX_OK
    assert moe.status() == B.REFLEX_OK
    pairs = int(k_sum.item())
    rec = moe.record()
    counts = rec["counts"].cpu().numpy()
    step(p_fixed)
    torch.cuda.synchronize(dev)
    pairs_fixed = int(k_sum.item())

    # ---- timed region: REFLEX counts, one step per graph replay ----
    g_reflex = graph_of(lambda: step(p_reflex))
    ms = timed(g_reflex, args.steps, args.warmup)
    ms = max_over_ranks(ms)
    ms_step = ms / args.steps
    # ---- gate/up GEMM launches: the same step with events around the GEMM,
    # 16 steps per graph; the durations of the last replay are averaged ----
    NS = 16
    try:   # timestamps recorded by graph nodes need external event records
        up_evs = [[torch.cuda.Event(enable_timing=True, external=True) for _ in range(2)]
                  for _ in range(NS)]

        def staged_block():
            for e in up_evs:
                staged_step(p_reflex, e)
        timed(graph_of(staged_block), max(1, min(args.steps, 400) // NS), 1)
    except TypeError:  # older torch: the same staged steps, launched eagerly
        up_evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(NS)]
        for _ in range(2):
            for e in up_evs:
                staged_step(p_reflex, e)
        barrier()
    up_times = [e[0].elapsed_time(e[1]) for e in up_evs]
    # ---- same kernels at fixed top-K_base ----
    g_fixed = graph_of(lambda: step(p_fixed))
    n_fixed = max(1, args.steps // 2)
    ms_fixed = max_over_ranks(timed(g_fixed, n_fixed, 2)) / n_fixed

    # ---- end to end from pinned host buffers: every step uploads its inputs
    # (hidden states and per-token state) and reads its output back.  Copies
    # run on a copy stream with two buffer sets, so the upload of step i+1 and
    # the read-back of step i-1 overlap the kernels of step i ----
    host_in = {k: torch.from_numpy(np.ascontiguousarray(v)).pin_memory()
               for k, v in state.items()}
    host_h = torch.from_numpy(np.ascontiguousarray(layer["hidden"]).view(
        np.int16 if cfg.dtype == "bf16" else np.float32)).pin_memory()
    host_out = [torch.empty((T, d), dtype=moe.tdtype).pin_memory() for _ in range(2)]
    dev_state = [{k: torch.empty_like(v) for k, v in ds.items()} for _ in range(2)]
    dev_h = [torch.empty_like(dl["hidden"]) for _ in range(2)]
    dev_out = [torch.empty_like(out) for _ in range(2)]
    h2d = sum(int(v.numel() * v.element_size()) for v in host_in.values()) + \
        int(host_h.numel() * host_h.element_size())
    d2h = int(host_out[0].numel() * host_out[0].element_size())
    copy_s = torch.cuda.Stream(dev)
    ev_up = [torch.cuda.Event() for _ in range(2)]
    ev_done = [torch.cuda.Event() for _ in range(2)]
    ev_read = [torch.cuda.Event() for _ in range(2)]

    def e2e_run(n: int):
        for i in range(n + 1):
            b = i & 1
            if i < n:
                with torch.cuda.stream(copy_s):   # upload step i
                    copy_s.wait_event(ev_done[b])  # step i-2 finished with buffer b
                    for k, v in host_in.items():
                        dev_state[b][k].copy_(v, non_blocking=True)
                    dev_h[b].view(host_h.dtype).copy_(host_h, non_blocking=True)
                    ev_up[b].record(copy_s)
                stream.wait_event(ev_up[b])
                stream.wait_event(ev_read[b])      # read-back of step i-2 done
                moe.step(dev_state[b], p_reflex, dev_h[b], out=dev_out[b], k_out=k_buf,
                         k_sum=k_sum, status=st, flags=F)
                ev_done[b].record(stream)
            if i > 0:
                pb = (i - 1) & 1
                with torch.cuda.stream(copy_s):   # read back step i-1
                    copy_s.wait_event(ev_done[pb])
                    host_out[pb].copy_(dev_out[pb], non_blocking=True)
                    ev_read[pb].record(copy_s)
        stream.wait_event(ev_read[(n - 1) & 1])

    e2e_run(max(3, args.warmup // 2))
    barrier()
    n_e2e = max(3, args.steps // 2)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    copy_s.wait_event(e0)
    e2e_run(n_e2e)
    e1.record(stream)
    barrier()
    ms_e2e = max_over_ranks(e0.elapsed_time(e1)) / n_e2e
    clocks = clk.stop()
    # the end-to-end outputs are those of the resident-input step, bit for bit
    g_reflex.replay()
    torch.cuda.synchronize(dev)
    assert torch.equal(host_out[(n_e2e - 1) & 1], out.cpu())

    if rank != 0:
        return
    peaks = load_peaks()
    tokens_per_s = R.whole_job_rate(T, world, ms_step)
    flops_step = 6.0 * d * I * pairs          # Eq. 10, routed experts
    # dominant kernel: grouped gate/up GEMM; algorithmic bytes per launch =
    # gate/up weights of the experts that received pairs + gathered rows read
    # + activations written (bf16)
    es = 2 if cfg.dtype == "bf16" else 4
    touched = int((counts > 0).sum())
    up_bytes = touched * 2 * I * d * es + pairs * d * es + pairs * I * es
    if S:
        up_bytes += 2 * S * d * es + T * d * es + T * S * es
    up_flops = 4.0 * pairs * d * I + (4.0 * T * d * S if S else 0.0)
    up_ms = statistics.mean(up_times) if up_times else float("nan")
    achieved_gbs = up_bytes / (up_ms * 1e-3) / 1e9
    hbm_bound = up_bytes / (peaks["hbm"] * 1e9) >= up_flops / (peaks["bf16"] * 1e12)
    if hbm_bound:
        roof = dict(bound="hbm", achieved=achieved_gbs, peak=peaks["hbm"],
                    unit="GB/s", frac=achieved_gbs / peaks["hbm"])
    else:
        tf = up_flops / (up_ms * 1e-3) / 1e12
        roof = dict(bound="tensor", achieved=tf, peak=peaks["bf16"],
                    unit="TFLOP/s", frac=tf / peaks["bf16"])
    roof.update(kernel="grouped_gemm_kernel, gate/up + SwiGLU (tcgen05)",
                traffic=ncu_traffic(cfg.name), algorithmic_bytes=up_bytes,
                algorithmic_flops=up_flops, avg_launch_ms=up_ms,
                peak_source=peaks["source"] + " (burst)")
    # layer roofline: all expert weights touched + hidden in/out vs Eq. 10 flops
    layer_bytes = touched * 3 * I * d * es + 2 * T * d * es + E * d * es
    if S:
        layer_bytes += 3 * S * d * es
    layer_flops = flops_step + (6.0 * d * S * T if S else 0.0)
    t_roof = max(layer_bytes / (peaks["hbm"] * 1e9), layer_flops / (peaks["bf16"] * 1e12))
    launches_per_step = api.step_launches(cfg.dtype, T, d, E, S, F)
    line = dict(
        metric=METRIC, value=tokens_per_s, unit="tokens/s",
        n_gpus=world, steps=args.steps, warmup=args.warmup, ms_per_step=ms_step,
        higher_is_better=True, scaling="weak", vs_baseline=None, dtype="bf16"
        if cfg.dtype == "bf16" else "f32", data="synthetic",
        config=dict(layer_config(cfg, world),
                    timing="CUDA-graph replay of one step (one reflex_step call: "
                           "allocation + forward) per "
                           "timed iteration; e2e: eager API calls, each step's upload "
                           "and read-back from pinned host memory on a copy stream, "
                           "double-buffered so they overlap the neighbouring steps"),
        expert_tflops=flops_step * world / (ms_step * 1e-3) / 1e12,
        # Eq. 10 counts the routed experts only; the shared expert's dense
        # SwiGLU (6 d s T) is added here
        expert_tflops_with_shared=(layer_flops * world / (ms_step * 1e-3) / 1e12
                                   if S else None),
        layer_roofline_frac=t_roof / (ms_step * 1e-3),
        avg_k=pairs / T, pairs=pairs,
        fixed_topk=dict(k=cfg.k_base, pairs=pairs_fixed, ms_per_step=ms_fixed,
                        value=R.whole_job_rate(T, world, ms_fixed),
                        expert_tflops=6.0 * d * I * pairs_fixed * world / (ms_fixed * 1e-3) / 1e12),
        roofline=roof,
        e2e=dict(value=R.whole_job_rate(T, world, ms_e2e), unit="tokens/s",
                 h2d_bytes_per_step=h2d, d2h_bytes_per_step=d2h,
                 ms_per_step=ms_e2e),
        gpu_launches=launches_per_step * args.steps,
        clocks=clocks,
    )
    if not args.no_cpu_baseline and world == 1:
        rate, n, dt, cores = oracle_rate(cfg, layer, state, args.cpu_seconds, seed)
        rate1, n1, dt1, _ = oracle_rate(cfg, layer, state, args.cpu_seconds / 2, seed + 1, 1)
        line["cpu_baseline"] = dict(
            value=rate, unit="tokens/s", cores=cores, kind="oracle",
            sample=f"{n} seeded tokens of the {T}-token batch, full oracle path "
                   f"(allocation on the whole batch), {dt:.1f} s",
            single_thread=dict(value=rate1, unit="tokens/s", cores=1,
                               sample=f"{n1} seeded tokens, {dt1:.1f} s"))
    elif world > 1:
        line["cpu_baseline"] = None
    if args.gather_in_gemm:
        line["dispatch"] = "rows gathered inside the gate/up GEMM (REFLEX_FLAG_GATHER_IN_GEMM)"
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# 16-layer stack (GPU): the default workload
# ---------------------------------------------------------------------------
STACK_LAYERS = 16
STACK_LAYER_CFG = "llada_moe_b32"


def stack_config(world: int) -> dict:
    cfg = W.CONFIGS[STACK_LAYER_CFG]
    return dict(workload="llada_moe_stack16",
                description=f"full denoising forward of {STACK_LAYERS} LLaDA-MoE-shaped "
                            f"layers (d=2048, E=64 SwiGLU experts, inter=1024, K in "
                            f"[2,12]), batch 32 x 1024 tokens (512 prompt + 512 gen, "
                            f"block 32), counts allocated once per forward and shared by "
                            f"every layer, residual h <- bf16(h + MoE(h)), fresh router "
                            f"and expert weights per layer, bf16 storage, fp32 "
                            f"accumulation",
                tokens_per_step=cfg.T, layers=STACK_LAYERS, parallelism=f"replicas{world}",
                l2="no flush: 12.9 GB of expert weights stream from HBM every step")


def oracle_stack(cfg, stack, state, tokens):
    """The oracle's whole forward for the listed tokens: the counts of the
    whole batch (Eq. 5 / Eq. 9 + clip; an active block couples its tokens),
    then every layer on those tokens (scores, TopK / alpha, pair order,
    Eq. 2, residual).  Tokens are independent across the layers (no
    attention), so the sample is exact."""
    import oracle
    k = oracle.allocate(state["conf1"], state["conf2"], state["hist_len"],
                        state["masked"], state["block_id"], state["seq_offsets"],
                        state["active_block"], **cfg.alloc_params())
    trace = oracle.moe_stack(stack["hidden"][tokens], stack["layers"], k[tokens],
                             cfg.k_max)
    return trace[-1]["h_out"]


def oracle_stack_rate(cfg, stack, state, target_s, seed, threads=None):
    """tokens/s (whole forwards) of the oracle on a seeded token sample sized to
    about target_s seconds; threads = None keeps the OpenMP default (all
    cores)."""
    import oracle
    oracle.build()
    all_cores = oracle.num_threads()
    if threads is not None:
        oracle.set_num_threads(threads)
    try:
        used = oracle.num_threads()
        T = stack["hidden"].shape[0]
        rng = np.random.default_rng(seed)
        n = max(2, min(T, 2 * used))
        t0 = time.perf_counter()
        oracle_stack(cfg, stack, state, np.sort(rng.choice(T, n, replace=False)).astype(np.int32))
        dt = time.perf_counter() - t0
        n2 = int(min(T, max(n, n * target_s / max(dt, 1e-6))))
        toks = np.sort(rng.choice(T, n2, replace=False)).astype(np.int32)
        t0 = time.perf_counter()
        oracle_stack(cfg, stack, state, toks)
        dt = time.perf_counter() - t0
    finally:
        oracle.set_num_threads(all_cores)
    return n2 / dt, n2, dt, used


def run_stack_reference(args, rank, world):
    """The oracle as it stands on the host cores, on the stack workload.  One
    token through the 16 layers costs about 0.5 core-seconds in the oracle,
    so a step samples (token, layer) units instead of whole tokens: an
    untimed oracle pass over a seeded pool of tokens records every layer's
    input, and each step computes the counts of the whole batch (Eq. 5 /
    Eq. 9 + clip) and then takes one seeded layer through n seeded pooled
    tokens (scores, TopK / alpha, pair order, Eq. 2, residual) on their
    inputs at that layer, in one call so that the host threads share it.
    Every layer has the same shapes, so n units are n / 16 whole forwards; n
    is sized so that the W + K steps take about two minutes."""
    import torch  # noqa: F401  (keeps the launch environment identical)
    if rank != 0:
        return
    import oracle
    oracle.build()
    cfg = W.CONFIGS[STACK_LAYER_CFG]
    L = STACK_LAYERS
    stack = W.make_stack(cfg, args.seed, L)
    state = W.make_state(cfg, args.seed)
    T = cfg.T
    rng = np.random.default_rng(args.seed)
    threads = oracle.num_threads()
    pool = np.sort(rng.choice(T, min(T, max(64, 16 * threads)), replace=False)).astype(np.int32)
    P = pool.size

    def counts():
        return oracle.allocate(state["conf1"], state["conf2"], state["hist_len"],
                               state["masked"], state["block_id"], state["seq_offsets"],
                               state["active_block"], **cfg.alloc_params())
    k_pool = counts()[pool]
    trace = oracle.moe_stack(stack["hidden"][pool], stack["layers"], k_pool, cfg.k_max)
    h_in = [trace[l]["h_in"] for l in range(L)]
    del trace

    def one(n):
        k_all = counts()
        l = int(rng.integers(L))
        ps = np.sort(rng.choice(P, n, replace=False))
        w = stack["layers"][l]
        res = oracle.moe_layer(h_in[l][ps], w["w_router"], w["w_gate_up"], w["w_down"],
                               k_all[pool[ps]], cfg.k_max)
        oracle.residual_bf16(h_in[l][ps], res["out"])

    per_step_s = min(5.0, 120.0 / max(1, args.steps + args.warmup))
    n0 = min(P, 4 * threads)
    t0 = time.perf_counter()
    one(n0)
    dt0 = time.perf_counter() - t0
    n = int(min(P, max(1, n0 * per_step_s / max(dt0, 1e-6))))
    for _ in range(args.warmup):
        one(n)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        one(n)
    dt = time.perf_counter() - t0
    value = n / L * args.steps / dt
    sample = (f"per step one seeded layer of {L} through {n} seeded tokens of a pool "
              f"of {P} from the {T}-token batch, on their inputs at that layer (from "
              f"an untimed oracle pass), plus the whole batch's counts: {n} / {L} "
              f"whole forwards per step")
    line = dict(metric=METRIC, value=value, unit="tokens/s", impl="reference",
                n_gpus=args.gpus, steps=args.steps, warmup=args.warmup,
                ms_per_step=1e3 * dt / args.steps, higher_is_better=True,
                scaling="weak", vs_baseline=None, dtype="f64", data="synthetic",
                config=stack_config(world),
                cpu_baseline=dict(value=value, unit="tokens/s", kind="oracle",
                                  cores=threads, sample=sample),
                e2e=dict(value=value, unit="tokens/s", h2d_bytes_per_step=0,
                         d2h_bytes_per_step=0))
    print(json.dumps(line), flush=True)


def run_stack(args, rank, world, local_rank):
    import torch
    from paper_2608_01784_gb300 import _binding as B
    from paper_2608_01784_gb300 import api, build

    build.build()
    B.load()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    cfg = W.CONFIGS[STACK_LAYER_CFG]
    L = STACK_LAYERS
    seed = R.rank_seed(args.seed, rank)
    T, d, E, I, km = cfg.T, cfg.d, cfg.E, cfg.inter, cfg.k_max
    # seeded host inputs (the oracle sees the same bits), then on the device
    stack = W.make_stack(cfg, seed, L)
    state = W.make_state(cfg, seed)
    ds = api.state_to_device(state, dev)
    layers = [api.layer_to_device(w, cfg.dtype, dev) for w in stack["layers"]]
    h0 = api.layer_to_device({"hidden": stack["hidden"]}, cfg.dtype, dev)["hidden"]
    net = api.MoEStack(layers, dtype=cfg.dtype, d=d, E=E, inter=I, shared_inter=0,
                       k_max=km, max_tokens=T, device=dev)
    stream = torch.cuda.current_stream(dev)
    k_buf = torch.empty(T, dtype=torch.int32, device=dev)
    k_sum = torch.zeros(1, dtype=torch.int64, device=dev)
    st = torch.zeros(1, dtype=torch.int32, device=dev)
    out = torch.empty_like(h0)
    F = B.REFLEX_FLAG_RENORM_TOPK | (B.REFLEX_FLAG_GATHER_IN_GEMM if args.gather_in_gemm else 0)
    p_reflex = B.make_params(**cfg.alloc_params())
    p_fixed = B.make_params(**cfg.alloc_params(delta_role=0, delta_cur=0))

    def forward(params, hidden=h0, dst=out, state_=ds, around_up=None):
        net.forward(state_, params, hidden, dst, k_buf, k_sum, st, flags=F,
                    around_up=around_up)

    def graph_of(fn):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, capture_error_mode="relaxed"):
            fn()
        return g

    def barrier():
        R.barrier(world, dev)

    def timed(graph, replays, warmup):
        for _ in range(warmup):
            graph.replay()
        barrier()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(replays):
            graph.replay()
        b.record(stream)
        barrier()
        return a.elapsed_time(b)

    clk = ClockSampler(local_rank)
    clk.start()
    # correctness gate before timing: counts and statuses clean
    forward(p_reflex)
    torch.cuda.synchronize(dev)
    assert B.reflex_read_status(st) == B.REFLEX_OK and net.status() == B.REFLEX_OK
    pairs = int(k_sum.item())
    forward(p_fixed)
    torch.cuda.synchronize(dev)
    assert net.status() == B.REFLEX_OK
    pairs_fixed = int(k_sum.item())
    # the routing of the last layer: experts that received pairs
    counts = net.moe.record()["counts"].cpu().numpy()

    # ---- timed region: one whole forward (counts + 16 layers) per replay ----
    g_reflex = graph_of(lambda: forward(p_reflex))
    ms = R.max_over_ranks(timed(g_reflex, args.steps, args.warmup), world, dev)
    ms_step = ms / args.steps
    # ---- gate/up GEMM launches: the same forward with events around every
    # layer's gate/up GEMM, in one graph; durations of the last replay ----
    try:   # timestamps recorded by graph nodes need external event records
        up_evs = [[torch.cuda.Event(enable_timing=True, external=True) for _ in range(2)]
                  for _ in range(L)]
        around = (lambda l: up_evs[l][0].record(), lambda l: up_evs[l][1].record())
        timed(graph_of(lambda: forward(p_reflex, around_up=around)), 2, 1)
    except TypeError:  # older torch: the same staged forward, launched eagerly
        up_evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(L)]
        around = (lambda l: up_evs[l][0].record(), lambda l: up_evs[l][1].record())
        for _ in range(2):
            forward(p_reflex, around_up=around)
        barrier()
    up_times = [e[0].elapsed_time(e[1]) for e in up_evs]
    # ---- same kernels at fixed top-K_base ----
    g_fixed = graph_of(lambda: forward(p_fixed))
    n_fixed = max(1, args.steps // 2)
    ms_fixed = R.max_over_ranks(timed(g_fixed, n_fixed, 2), world, dev) / n_fixed

    # ---- end to end through the public API from pinned host buffers: every
    # forward uploads its hidden states and per-token state and reads its
    # output back; copies on a copy stream, two buffer sets, so the upload of
    # forward i+1 and the read-back of forward i-1 overlap forward i ----
    host_in = {k: torch.from_numpy(np.ascontiguousarray(v)).pin_memory()
               for k, v in state.items()}
    host_h = torch.from_numpy(np.ascontiguousarray(stack["hidden"]).view(np.int16)).pin_memory()
    host_out = [torch.empty((T, d), dtype=torch.bfloat16).pin_memory() for _ in range(2)]
    dev_state = [{k: torch.empty_like(v) for k, v in ds.items()} for _ in range(2)]
    dev_h = [torch.empty_like(h0) for _ in range(2)]
    dev_out = [torch.empty_like(out) for _ in range(2)]
    h2d = sum(int(v.numel() * v.element_size()) for v in host_in.values()) + \
        int(host_h.numel() * host_h.element_size())
    d2h = int(host_out[0].numel() * host_out[0].element_size())
    copy_s = torch.cuda.Stream(dev)
    ev_up = [torch.cuda.Event() for _ in range(2)]
    ev_done = [torch.cuda.Event() for _ in range(2)]
    ev_read = [torch.cuda.Event() for _ in range(2)]

    def e2e_run(n: int):
        for i in range(n + 1):
            b = i & 1
            if i < n:
                with torch.cuda.stream(copy_s):   # upload forward i
                    copy_s.wait_event(ev_done[b])  # forward i-2 finished with set b
                    for k, v in host_in.items():
                        dev_state[b][k].copy_(v, non_blocking=True)
                    dev_h[b].view(torch.int16).copy_(host_h, non_blocking=True)
                    ev_up[b].record(copy_s)
                stream.wait_event(ev_up[b])
                stream.wait_event(ev_read[b])      # read-back of forward i-2 done
                forward(p_reflex, hidden=dev_h[b], dst=dev_out[b], state_=dev_state[b])
                ev_done[b].record(stream)
            if i > 0:
                pb = (i - 1) & 1
                with torch.cuda.stream(copy_s):   # read back forward i-1
                    copy_s.wait_event(ev_done[pb])
                    host_out[pb].copy_(dev_out[pb], non_blocking=True)
                    ev_read[pb].record(copy_s)
        stream.wait_event(ev_read[(n - 1) & 1])

    e2e_run(2)
    barrier()
    n_e2e = max(3, args.steps // 2)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    copy_s.wait_event(e0)
    e2e_run(n_e2e)
    e1.record(stream)
    barrier()
    ms_e2e = R.max_over_ranks(e0.elapsed_time(e1), world, dev) / n_e2e
    clocks = clk.stop()
    # the end-to-end outputs are those of the resident-input forward, bit for bit
    g_reflex.replay()
    torch.cuda.synchronize(dev)
    assert torch.equal(host_out[(n_e2e - 1) & 1], out.cpu())
    assert net.status() == B.REFLEX_OK

    if rank != 0:
        return
    peaks = load_peaks()
    flops_layer = 6.0 * d * I * pairs                  # Eq. 10, routed experts
    # dominant kernel: the CTA-pair gate/up (SwiGLU) GEMM, tensor-bound on
    # this shape; algorithmic FLOPs per launch = 4 d inter sum(k); it runs
    # inside a ~30 ms forward, so the sustained bf16 peak is the denominator
    up_flops = 4.0 * pairs * d * I
    touched = int((counts > 0).sum())
    up_bytes = touched * 2 * I * d * 2 + pairs * d * 2 + pairs * I * 2
    up_ms = statistics.mean(up_times)
    tf = up_flops / (up_ms * 1e-3) / 1e12
    peak_sus = peaks["bf16_sustained"] or peaks["bf16"]
    roof = dict(bound="tensor", achieved=tf, peak=peak_sus, unit="TFLOP/s",
                frac=tf / peak_sus, traffic=ncu_traffic("llada_moe_stack16"),
                kernel="grouped_gemm_pair_kernel<0>: gate/up + SwiGLU, cta_group::2 "
                       "tcgen05, TMEM accumulators, TMA-fed",
                algorithmic_flops=up_flops, algorithmic_bytes=up_bytes,
                avg_launch_ms=up_ms, launches_averaged=len(up_times),
                frac_of_burst=tf / peaks["bf16"],
                peak_source=peaks["source"] + " (sustained bf16; the kernel runs "
                                              "inside a long step)")
    launches = 1 + L * (api.step_launches(cfg.dtype, T, d, E, 0, F) - 1)
    line = dict(
        metric=METRIC, value=R.whole_job_rate(T, world, ms_step), unit="tokens/s",
        n_gpus=world, steps=args.steps, warmup=args.warmup, ms_per_step=ms_step,
        higher_is_better=True, scaling="weak", vs_baseline=None, dtype="bf16",
        data="synthetic",
        config=dict(stack_config(world),
                    timing="CUDA-graph replay of one whole forward (counts + 16 "
                           "layers) per timed iteration; e2e: eager API calls, each "
                           "forward's upload and read-back from pinned host memory on a "
                           "copy stream, double-buffered"),
        expert_tflops=flops_layer * L * world / (ms_step * 1e-3) / 1e12,
        expert_frac_of_bf16_sustained=flops_layer * L / (ms_step * 1e-3) / 1e12 / peak_sus,
        avg_k=pairs / T, pairs_per_layer=pairs,
        fixed_topk=dict(k=cfg.k_base, pairs_per_layer=pairs_fixed, ms_per_step=ms_fixed,
                        value=R.whole_job_rate(T, world, ms_fixed),
                        expert_tflops=6.0 * d * I * pairs_fixed * L * world
                        / (ms_fixed * 1e-3) / 1e12),
        roofline=roof,
        e2e=dict(value=R.whole_job_rate(T, world, ms_e2e), unit="tokens/s",
                 h2d_bytes_per_step=h2d, d2h_bytes_per_step=d2h, ms_per_step=ms_e2e,
                 api="MoEStack.forward: reflex_step (counts + layer 0), then "
                     "reflex_moe_forward per layer"),
        gpu_launches=launches * args.steps,
        clocks=clocks,
    )
    if not args.no_cpu_baseline and world == 1:
        budget = args.cpu_seconds
        rate, n, dt, cores = oracle_stack_rate(cfg, stack, state, budget, seed)
        rate1, n1, dt1, _ = oracle_stack_rate(cfg, stack, state, budget / 2, seed + 1, 1)
        line["cpu_baseline"] = dict(
            value=rate, unit="tokens/s", cores=cores, kind="oracle",
            sample=f"{n} seeded tokens of the {T}-token batch through all {L} layers "
                   f"(counts on the whole batch; tokens are independent across "
                   f"layers), {dt:.1f} s, rate per whole forward",
            single_thread=dict(value=rate1, unit="tokens/s", cores=1,
                               sample=f"{n1} seeded tokens, {dt1:.1f} s"))
    elif world > 1:
        line["cpu_baseline"] = None
    if args.gather_in_gemm:
        line["dispatch"] = "rows gathered inside the gate/up GEMM (REFLEX_FLAG_GATHER_IN_GEMM)"
    print(json.dumps(line), flush=True)


def run_sweep(args, rank, world, local_rank):
    import torch
    from paper_2608_01784_gb300 import _binding as B
    from paper_2608_01784_gb300 import api, build

    build.build()
    B.load()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    cfg = W.CONFIGS["llada2_mini"]
    if args.sweep_tokens:
        tokens = [int(x) for x in args.sweep_tokens.split(",")]
    else:
        tokens = [256 << i for i in range(9)]          # 256 .. 65536
    skews = ([float(x) for x in args.sweep_skews.split(",")] if args.sweep_skews
             else [0.0, 0.25, 0.5, 0.75, 1.0])
    if min(tokens) < 1 or not skews:
        raise SystemExit("--sweep-tokens and --sweep-skews need positive values")
    Tmax = max(tokens)
    d, E, I, S, km = cfg.d, cfg.E, cfg.inter, cfg.shared_inter, cfg.k_max
    layer = W.make_layer(cfg, args.seed, T=Tmax)
    dl = api.layer_to_device(layer, cfg.dtype, dev)
    moe = api.MoELayer(dl, dtype=cfg.dtype, d=d, E=E, inter=I, shared_inter=S,
                       k_max=km, max_tokens=Tmax, device=dev)
    stream = torch.cuda.current_stream(dev)
    peaks = load_peaks()
    F = B.REFLEX_FLAG_RENORM_TOPK
    for T in tokens:
        h = dl["hidden"][:T]
        out = torch.empty((T, d), dtype=moe.tdtype, device=dev)
        base_ms = None
        for skew in skews:
            k = torch.from_numpy(W.skewed_k(T, skew, cfg.k_min, cfg.k_base, km,
                                            seed=args.seed)).to(dev)
            moe.forward(h, k, out, F)
            torch.cuda.synchronize(dev)
            assert moe.status() == B.REFLEX_OK
            counts = moe.record()["counts"].cpu().numpy()
            pairs = int(counts.sum())
            steps = max(5, min(200, int(2e5 // T) + 5))
            for _ in range(3):
                moe.forward(h, k, out, F)
            torch.cuda.synchronize(dev)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for _ in range(steps):
                moe.forward(h, k, out, F)
            b.record(stream)
            torch.cuda.synchronize(dev)
            ms = a.elapsed_time(b) / steps
            if skew == 0.0:
                base_ms = ms
            touched = int((counts > 0).sum())
            bytes_ = (touched * 3 * I * d + 3 * S * d + 2 * T * d + E * d) * 2
            flops = 6.0 * d * I * pairs + 6.0 * d * S * T
            t_roof = max(bytes_ / (peaks["hbm"] * 1e9), flops / (peaks["bf16"] * 1e12))
            line = dict(sweep="llada2_mini", tokens=T, skew=skew, avg_k=pairs / T,
                        pairs=pairs, ms=ms, tokens_per_s=T / (ms * 1e-3),
                        expert_tflops=6.0 * d * I * pairs / (ms * 1e-3) / 1e12,
                        expert_tflops_with_shared=flops / (ms * 1e-3) / 1e12,
                        roofline_frac=t_roof / (ms * 1e-3),
                        bound="hbm" if bytes_ / (peaks["hbm"] * 1e9) >= flops / (peaks["bf16"] * 1e12) else "tensor",
                        load_imbalance=float(counts.max() / max(counts.mean(), 1e-9)),
                        vs_uniform_kbase=ms / base_ms if base_ms else None)
            print(json.dumps(line), flush=True)


ABLATIONS = [  # (name, allocation overrides): REFLEX and its App. C ablations
    ("reflex", {}),
    ("rrb_only", dict(delta_cur=0)),
    ("fger_only", dict(delta_role=0)),
    ("role_shuffled_rrb", dict(delta_cur=0, role_shuffle=1)),
    ("frontier_only", dict(signal=1)),
    ("progress_only", dict(signal=2)),
    ("confidence_only", dict(signal=3)),
    ("uncertainty_only", dict(signal=4)),
    ("fixed_topk", dict(delta_role=0, delta_cur=0)),
]
# The threshold-based comparison methods of App. B on the same kernels (count
# bounds [1, 12]; low / high thresholds per model family as the paper sets
# them): Top-p mass p and the Expert-Threshold router weight.
RULE_SETTINGS = {
    "llada_moe": dict(top_p=(0.15, 0.20), expert_thr=(0.0215, 0.0190)),
    "llada_moe_b32": dict(top_p=(0.15, 0.20), expert_thr=(0.0215, 0.0190)),
    "llada2_mini": dict(top_p=(0.25, 0.325), expert_thr=(0.0270, 0.0220)),
}


def rule_ablations(cfg_name: str):
    r = RULE_SETTINGS.get(cfg_name)
    if r is None:
        return []
    out = []
    for tag, v in zip(("low", "high"), r["top_p"]):
        out.append((f"top_p_{tag}", dict(count_rule=1, rule_threshold=v, k_min=1, k_max=12)))
    for tag, v in zip(("low", "high"), r["expert_thr"]):
        out.append((f"expert_threshold_{tag}",
                    dict(count_rule=2, rule_threshold=v, k_min=1, k_max=12)))
    return out


def run_ablation(args, rank, world, local_rank):
    """One JSON line per allocation variant on the same layer and state:
    realised counts (avg k, pairs), the allocation kernel's own time and the
    whole step (allocation + layer).  The role shuffle draws a new seed every
    step (one permutation per denoising forward)."""
    import torch
    from paper_2608_01784_gb300 import _binding as B
    from paper_2608_01784_gb300 import api, build

    build.build()
    B.load()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    cfg = W.CONFIGS.get(args.config, W.CONFIGS["llada_moe"])
    T, d, E, I, S, km = cfg.T, cfg.d, cfg.E, cfg.inter, cfg.shared_inter, cfg.k_max
    dl = api.layer_to_device(W.make_layer(cfg, args.seed), cfg.dtype, dev)
    ds = api.state_to_device(W.make_state(cfg, args.seed), dev)
    moe = api.MoELayer(dl, dtype=cfg.dtype, d=d, E=E, inter=I, shared_inter=S,
                       k_max=km, max_tokens=T, device=dev)
    stream = torch.cuda.current_stream(dev)
    k_buf = torch.empty(T, dtype=torch.int32, device=dev)
    k_sum = torch.zeros(1, dtype=torch.int64, device=dev)
    st = torch.zeros(1, dtype=torch.int32, device=dev)
    out = torch.empty((T, d), dtype=moe.tdtype, device=dev)
    F = B.REFLEX_FLAG_RENORM_TOPK
    steps = max(20, min(args.steps, 500))

    def timed(fn):
        for i in range(3):
            fn(i)
        torch.cuda.synchronize(dev)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for i in range(steps):
            fn(i)
        b.record(stream)
        torch.cuda.synchronize(dev)
        return a.elapsed_time(b) / steps

    for name, over in ABLATIONS + rule_ablations(cfg.name):
        params = [B.make_params(**cfg.alloc_params(**over, shuffle_seed=args.seed + i))
                  for i in range(steps)]
        rule = over.get("count_rule", 0)
        scores = None
        if rule:   # the score rules' counts from the layer's own router scores
            moe.forward(dl["hidden"], k_buf, out, F | B.REFLEX_STAGE_ROUTE |
                        B.REFLEX_FLAG_EXACT_SCORES)
            scores = moe.record()["scores"].clone()

        def alloc(i):
            if rule:
                api.allocate(None, params[i % steps], E, stream, k_buf, k_sum, st,
                             router_scores=scores)
            else:
                api.allocate(ds, params[i % steps], E, stream, k_buf, k_sum, st)

        def step(i):
            moe.step(ds, params[i % steps], dl["hidden"], out=out, k_out=k_buf,
                     k_sum=k_sum, status=st, flags=F)

        alloc(0)
        moe.forward(dl["hidden"], k_buf, out, F)
        torch.cuda.synchronize(dev)
        assert B.reflex_read_status(st) == B.REFLEX_OK and moe.status() == B.REFLEX_OK
        pairs = int(k_sum.item())
        ms_alloc = timed(alloc)
        ms = timed(step)
        line = dict(ablation=name, workload=cfg.name, tokens=T, avg_k=pairs / T,
                    pairs=pairs, alloc_us=1e3 * ms_alloc, ms_per_step=ms,
                    count_rule=("reflex" if not rule else
                                "top_p" if rule == 1 else "expert_threshold"),
                    rule_threshold=over.get("rule_threshold"),
                    tokens_per_s=T / (ms * 1e-3),
                    expert_tflops=6.0 * d * I * pairs / (ms * 1e-3) / 1e12)
        print(json.dumps(line), flush=True)


def run_trajectory(args, rank, world, local_rank):
    """Whole denoising trajectories (allocation -> MoE layer -> state update per
    forward, from the all-mask start until every block is resolved) with the
    synthetic confidence model; one JSON line per workload and allocation:
    NFE, pairs per sample, AvgK and wall time."""
    import torch
    from paper_2608_01784_gb300 import _binding as B
    from paper_2608_01784_gb300 import api, build
    from paper_2608_01784_gb300 import trajectory as TR

    build.build()
    B.load()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    stream = torch.cuda.current_stream(dev)
    for name in ("llada_moe", "llada2_mini"):
        cfg = W.CONFIGS[name]
        dl = api.layer_to_device(W.make_layer(cfg, args.seed), cfg.dtype, dev)
        moe = api.MoELayer(dl, dtype=cfg.dtype, d=cfg.d, E=cfg.E, inter=cfg.inter,
                           shared_inter=cfg.shared_inter, k_max=cfg.k_max,
                           max_tokens=cfg.T, device=dev)
        st0 = TR.initial_state(W.make_state(cfg, args.seed))
        for alloc, over in (("reflex", {}), ("fixed_topk", dict(delta_role=0, delta_cur=0))):
            p = B.make_params(**cfg.alloc_params(**over))
            TR.simulate(api.state_to_device(st0, dev), p, cfg.E, seed=args.seed, moe=moe,
                        hidden=dl["hidden"], check_every=4, graph=True)  # warm-up run
            ds = api.state_to_device(st0, dev)
            torch.cuda.synchronize(dev)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            r = TR.simulate(ds, p, cfg.E, seed=args.seed, moe=moe, hidden=dl["hidden"],
                            check_every=4, graph=True)
            b.record(stream)
            torch.cuda.synchronize(dev)
            ms = a.elapsed_time(b)
            assert r["alloc_status"] == B.REFLEX_OK and r["update_status"] == B.REFLEX_OK
            lens = np.diff(st0["seq_offsets"])
            line = dict(trajectory=name, allocation=alloc, sequences=int(lens.size),
                        nfe_mean=float(r["nfe"].mean()), nfe_max=int(r["nfe"].max()),
                        forwards_run=r["forwards"],
                        pairs_per_sample=float(r["pairs"].mean()),
                        avg_k=float(r["pairs"].sum() / (r["nfe"] * lens).sum()),
                        ms_total=ms, ms_per_forward=ms / max(1, r["forwards"]),
                        samples_per_s=lens.size / (ms * 1e-3),
                        note="synthetic confidences; 1 MoE layer per forward; one "
                             "forward per CUDA-graph replay")
            print(json.dumps(line), flush=True)


def main():
    args = parse()
    ri = R.rank_info()
    world, rank, local_rank = ri.world, ri.rank, ri.local_rank
    # the GPU arm reduces on the GPUs (NCCL); the reference arm is host-only
    R.init(world, "nccl" if args.impl == "reflex" else "gloo", local_rank)
    stack = args.config == "llada_moe_stack16"
    try:
        if args.impl == "reference":
            if stack:
                run_stack_reference(args, rank, world)
            else:
                run_reference(args, W.CONFIGS[args.config], rank, world)
        elif args.sweep:
            if rank == 0:
                run_sweep(args, rank, world, local_rank)
        elif args.ablation:
            if rank == 0:
                run_ablation(args, rank, world, local_rank)
        elif args.trajectory:
            if rank == 0:
                run_trajectory(args, rank, world, local_rank)
        elif stack:
            run_stack(args, rank, world, local_rank)
        else:
            run_gpu(args, W.CONFIGS[args.config], rank, world, local_rank)
    finally:
        R.finalize(world)


if __name__ == "__main__":
    main()
