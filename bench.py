"""Benchmark of the REFLEX per-forward MoE hot path on GB300.

One step = one denoising forward's hot path on one batch, one reflex_step
call: the per-token counts of reflex_allocate (Eq. 5 / Eq. 9 + clip) and
reflex_moe_forward with them (router scores, variable-count TopK, pair
dispatch, grouped SwiGLU expert GEMMs on tcgen05, weighted combine; Eq. 2),
the count kernel running beside the router scores.
Default workload: the LLaDA-MoE-shaped layer (T = 1024 tokens: 512 prompt +
512 generated in blocks of 32; d = 2048, E = 64 SwiGLU experts with inter =
1024; K in [2, 12]; bf16 storage, fp32 accumulation), synthetic inputs.

Prints ONE JSON line (rank 0).  `value` = MoE-layer tokens/s over all ranks;
`expert_tflops` = 6 d inter sum(k) / step time (Eq. 10); the same kernels at
fixed top-K_base run beside it; `roofline` is for the dominant kernel, the
grouped gate/up (SwiGLU) GEMM; `e2e` times the same step from pinned host
buffers through the C ABI with the copies inside the timed region.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reflex|reference]
                  [--config NAME] [--no-cpu-baseline] [--sweep]
--config llada_moe_stack16: a whole denoising forward of 16 LLaDA-MoE-shaped
layers (batch 32 x 1024 tokens, counts allocated once and shared by every
layer, residual connection, fresh weights per layer drawn on the device).
--sweep: LLaDA2.0-mini layer shapes, 256 .. 65536 tokens x count skew
0 .. 1 (0 = uniform K_base, 1 = 70% K_min / 30% K_max), forward only.
Under torchrun each rank runs its own batch on its own GPU (weak scaling, no
data-path collective; a barrier and a max-reduce of the times only).
"""
from __future__ import annotations

import argparse
import json
import os
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

# DRAM bytes (read + write) moved per launch by the dominant kernel, from an
# ncu capture of the current kernel on the same workload
# (profiles/grouped_gemm_llada_moe_T1024.md,
# profiles/grouped_gemm_pair_llada2_mini_T8192.md); workloads without a
# capture of the current kernel report null.
NCU_TRAFFIC_BYTES = {"llada_moe": 561284352, "llada2_mini": 1407363048}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="reflex", choices=["reflex", "reference"])
    ap.add_argument("--config", default="llada_moe",
                    choices=sorted(W.CONFIGS) + ["llada_moe_stack16"])
    ap.add_argument("--sweep", action="store_true",
                    help="token-count x count-skew sweep on the LLaDA2.0-mini "
                         "layer (one JSON line per point)")
    ap.add_argument("--trajectory", action="store_true",
                    help="whole denoising trajectories: NFE and pairs per sample")
    ap.add_argument("--ablation", action="store_true",
                    help="REFLEX and its App. C allocation ablations on one layer")
    ap.add_argument("--seed", type=int, default=0)
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
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown",
                 "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return dict(sm_mhz=statistics.median(sm) if sm else None,
                    sm_max_mhz=max(mx) if mx else None,
                    reasons=sorted(reasons), samples=len(sm))


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


def oracle_rate(cfg, layer, state, target_s, seed=0):
    """tokens/s of the oracle on a seeded token sample sized to ~target_s."""
    import oracle
    oracle.build()
    T = layer["hidden"].shape[0]
    rng = np.random.default_rng(seed)
    n = min(T, 16)
    t0 = time.perf_counter()
    oracle_step(cfg, layer, state, np.sort(rng.choice(T, n, replace=False)).astype(np.int32))
    dt = time.perf_counter() - t0
    n2 = int(min(T, max(n, n * target_s / max(dt, 1e-6))))
    toks = np.sort(rng.choice(T, n2, replace=False)).astype(np.int32)
    t0 = time.perf_counter()
    oracle_step(cfg, layer, state, toks)
    dt = time.perf_counter() - t0
    return n2 / dt, n2, dt, oracle.num_threads()


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
                config=dict(workload=cfg.name, description=cfg.description,
                            tokens_per_step_sample=n),
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
    F = B.REFLEX_FLAG_RENORM_TOPK
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
    clk = ClockSampler(local_rank)
    clk.start()
    ms = timed(g_reflex, args.steps, args.warmup)
    clocks = clk.stop()
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
                traffic=NCU_TRAFFIC_BYTES.get(cfg.name), algorithmic_bytes=up_bytes,
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
        config=dict(workload=cfg.name, description=cfg.description,
                    tokens_per_step=T, parallelism=f"replicas{world}",
                    l2="no flush: expert weights > 129 MB L2 stream from HBM every step",
                    timing="CUDA-graph replay of one step (one reflex_step call: "
                           "allocation + forward) per "
                           "timed iteration; e2e: eager API calls, each step's upload "
                           "and read-back from pinned host memory on a copy stream, "
                           "double-buffered so they overlap the neighbouring steps"),
        expert_tflops=flops_step * world / (ms_step * 1e-3) / 1e12,
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
        clocks=dict(sm_mhz=clocks["sm_mhz"], sm_max_mhz=clocks["sm_max_mhz"],
                    reasons=clocks["reasons"], samples=clocks["samples"]),
    )
    if not args.no_cpu_baseline and world == 1:
        rate, n, dt, cores = oracle_rate(cfg, layer, state, args.cpu_seconds, seed)
        line["cpu_baseline"] = dict(
            value=rate, unit="tokens/s", cores=cores, kind="oracle",
            sample=f"{n} seeded tokens of the {T}-token batch, full oracle path "
                   f"(allocation on the whole batch), {dt:.1f} s")
    elif world > 1:
        line["cpu_baseline"] = None
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# 16-layer stack and sweep (GPU)
# ---------------------------------------------------------------------------
STACK_LAYERS = 16


def _device_weights(cfg, seed, dev, std):
    """Random-init bf16 weights of one layer drawn on the device (seeded)."""
    import torch
    g = torch.Generator(device=dev)
    g.manual_seed(int(seed))
    E, d, I = cfg.E, cfg.d, cfg.inter

    def rnd(*shape):
        return (torch.randn(*shape, generator=g, device=dev, dtype=torch.float32)
                * std).to(torch.bfloat16)
    return dict(w_router=rnd(E, d), w_gate_up=rnd(E, 2 * I, d), w_down=rnd(E, d, I))


def run_stack(args, rank, world, local_rank):
    import torch
    from paper_2608_01784_gb300 import _binding as B
    from paper_2608_01784_gb300 import api, build

    build.build()
    B.load()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    cfg = W.CONFIGS["llada_moe_b32"]
    seed = R.rank_seed(args.seed, rank)
    T, d, E, I, km = cfg.T, cfg.d, cfg.E, cfg.inter, cfg.k_max
    state = api.state_to_device(W.make_state(cfg, seed), dev)
    h0 = api.layer_to_device({"hidden": W.make_layer(cfg.with_(E=1, inter=64), seed)["hidden"]},
                             cfg.dtype, dev)["hidden"]
    layers = [_device_weights(cfg, 1000 * seed + l, dev, cfg.weight_std)
              for l in range(STACK_LAYERS)]
    # one workspace serves every layer (layers run one after another)
    moe = api.MoELayer(layers[0], dtype=cfg.dtype, d=d, E=E, inter=I, shared_inter=0,
                       k_max=km, max_tokens=T, device=dev)
    bufs = [torch.empty_like(h0), torch.empty_like(h0)]
    stream = torch.cuda.current_stream(dev)
    k_buf = torch.empty(T, dtype=torch.int32, device=dev)
    k_sum = torch.zeros(1, dtype=torch.int64, device=dev)
    st = torch.zeros(1, dtype=torch.int32, device=dev)
    F = B.REFLEX_FLAG_RENORM_TOPK | B.REFLEX_FLAG_RESIDUAL

    def forward(params):
        api.allocate(state, params, E, stream, k_buf, k_sum, st)
        h = h0
        for l, w in enumerate(layers):
            moe.w = w
            moe.forward(h, k_buf, bufs[l & 1], F)
            h = bufs[l & 1]

    def timed(params, steps, warmup):
        for _ in range(warmup):
            forward(params)
        R.barrier(world, dev)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(steps):
            forward(params)
        b.record(stream)
        R.barrier(world, dev)
        return R.max_over_ranks(a.elapsed_time(b) / steps, world, dev)

    p_reflex = B.make_params(**cfg.alloc_params())
    p_fixed = B.make_params(**cfg.alloc_params(delta_role=0, delta_cur=0))
    forward(p_reflex)
    torch.cuda.synchronize(dev)
    assert B.reflex_read_status(st) == B.REFLEX_OK and moe.status() == B.REFLEX_OK
    pairs = int(k_sum.item())
    forward(p_fixed)
    torch.cuda.synchronize(dev)
    pairs_fixed = int(k_sum.item())
    clk = ClockSampler(local_rank)
    clk.start()
    ms = timed(p_reflex, args.steps, args.warmup)
    clocks = clk.stop()
    ms_fixed = timed(p_fixed, max(1, args.steps // 2), 2)
    if rank != 0:
        return
    peaks = load_peaks()
    L = STACK_LAYERS
    flops = 6.0 * d * I * pairs * L
    flops_fixed = 6.0 * d * I * pairs_fixed * L
    line = dict(
        metric=METRIC, value=R.whole_job_rate(T, world, ms), unit="tokens/s", n_gpus=world,
        steps=args.steps, warmup=args.warmup, ms_per_step=ms, higher_is_better=True,
        scaling="weak", vs_baseline=None, dtype="bf16", data="synthetic",
        config=dict(workload="llada_moe_stack16",
                    description=f"{L} LLaDA-MoE-shaped layers (d=2048, E=64, inter=1024), "
                                f"batch 32 x 1024 tokens, counts allocated once per forward, "
                                f"residual h <- h + MoE(h), weights drawn on the device",
                    tokens_per_step=T, layers=L, parallelism=f"replicas{world}",
                    l2="no flush: 12.9 GB of expert weights stream every step"),
        expert_tflops=flops * world / (ms * 1e-3) / 1e12,
        expert_frac_of_bf16_peak=flops / (ms * 1e-3) / 1e12 / peaks["bf16_sustained"],
        avg_k=pairs / T, pairs_per_layer=pairs,
        fixed_topk=dict(k=cfg.k_base, pairs_per_layer=pairs_fixed, ms_per_step=ms_fixed,
                        value=R.whole_job_rate(T, world, ms_fixed),
                        expert_tflops=flops_fixed * world / (ms_fixed * 1e-3) / 1e12),
        # the counts once, then every layer's forward
        gpu_launches=args.steps * (1 + L * (api.step_launches(cfg.dtype, T, d, E, 0, F) - 1)),
        clocks=dict(sm_mhz=clocks["sm_mhz"], sm_max_mhz=clocks["sm_max_mhz"],
                    reasons=clocks["reasons"], samples=clocks["samples"]),
        peak_source=peaks["source"] + " (sustained bf16, long step)")
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
    Tmax = 65536
    d, E, I, S, km = cfg.d, cfg.E, cfg.inter, cfg.shared_inter, cfg.k_max
    layer = W.make_layer(cfg, args.seed, T=Tmax)
    dl = api.layer_to_device(layer, cfg.dtype, dev)
    moe = api.MoELayer(dl, dtype=cfg.dtype, d=d, E=E, inter=I, shared_inter=S,
                       k_max=km, max_tokens=Tmax, device=dev)
    stream = torch.cuda.current_stream(dev)
    peaks = load_peaks()
    F = B.REFLEX_FLAG_RENORM_TOPK
    T = 256
    while T <= Tmax:
        h = dl["hidden"][:T]
        out = torch.empty((T, d), dtype=moe.tdtype, device=dev)
        base_ms = None
        for skew in (0.0, 0.25, 0.5, 0.75, 1.0):
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
                        roofline_frac=t_roof / (ms * 1e-3),
                        bound="hbm" if bytes_ / (peaks["hbm"] * 1e9) >= flops / (peaks["bf16"] * 1e12) else "tensor",
                        load_imbalance=float(counts.max() / max(counts.mean(), 1e-9)),
                        vs_uniform_kbase=ms / base_ms)
            print(json.dumps(line), flush=True)
        T *= 2


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

    for name, over in ABLATIONS:
        params = [B.make_params(**cfg.alloc_params(**over, shuffle_seed=args.seed + i))
                  for i in range(steps)]

        def alloc(i):
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
    cfg = W.CONFIGS.get(args.config, W.CONFIGS["llada_moe_b32"])
    ri = R.rank_info()
    world, rank, local_rank = ri.world, ri.rank, ri.local_rank
    # the GPU arm reduces on the GPUs (NCCL); the reference arm is host-only
    R.init(world, "nccl" if args.impl == "reflex" else "gloo", local_rank)
    try:
        if args.impl == "reference":
            run_reference(args, cfg, rank, world)
        elif args.sweep:
            if rank == 0:
                run_sweep(args, rank, world, local_rank)
        elif args.ablation:
            if rank == 0:
                run_ablation(args, rank, world, local_rank)
        elif args.trajectory:
            if rank == 0:
                run_trajectory(args, rank, world, local_rank)
        elif args.config == "llada_moe_stack16":
            run_stack(args, rank, world, local_rank)
        else:
            run_gpu(args, cfg, rank, world, local_rank)
    finally:
        R.finalize(world)


if __name__ == "__main__":
    main()
