"""Benchmark of the tq2_0_fx4 MoE decode hot path on GB300.

Workload (one "step" = one token through one routed-expert MoE layer): 256
experts with gate/up 4096 -> 2048 and down 2048 -> 4096 projections in
tq2_0_fx4 (Student-t(5) * 0.02 synthetic weights, 3.27 GB of blocks), an
N(0, 0.02) fp32 router, top-8 with renormalized weights, N(0, 1) hidden
states. Every step routes a different hidden state, so the experts it reads
are (almost always) not the previous step's: the 3.27 GB expert pool is
larger than the 129 MB L2.

Metric: effective tq2_0_fx4 GB/s = (bytes of the 8 selected experts' blocks +
router weights) per token / time per token; tokens/s per MoE layer is the
same number divided by the bytes per token, reported beside it.

    python bench.py [--steps K] [--warmup W] [--gpus N] [--impl ours|reference]
                    [--workload moe_decode|gemv_1024|expert_ffn|grouped_decode_64|prefill_2048|
                                tiered_decode|mxfp4_gemv|moe_decode_mxfp4|free_gemv|pack_tied]

The K timed steps are captured once into a CUDA graph and replayed inside
the timed region (no host launch work in it); the other workloads time
tqfx4_moe_grouped on a batch of 64 tokens with Zipf(1.1) routing or 2048
tokens with uniform routing (tokens/s).

Under torchrun (N > 1) every rank runs its own replica on its own GPU (the
path has no exchange step here: replicas only) and rank 0 reports the
aggregate.
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

E, H, I, TOPK = 256, 4096, 2048, 8
SEED = 0
POOL = 256  # distinct hidden states cycled through the steps
WORKLOAD = "moe_decode_t1_e256_h4096_i2048_top8"
METRIC = "effective tq2_0_fx4 GB/s (MoE-layer decode)"
WORKLOAD_MX = "moe_decode_mxfp4_t1_e256_h4096_i2048_top8"
METRIC_MX = "effective MXFP4 GB/s (MoE-layer decode)"


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


# DRAM bytes (read + write) of one gate_up_kernel launch, from an ncu --set full capture of the
# 64-expert layer (one launch reads the 8 selected experts whatever the expert count). Set to None
# when the kernel changes until it is captured again.
GATE_UP_TRAFFIC = 68200448 + 936704
# The same for one tc_gemm_kernel gate/up launch of the 2048-token prefill: an ncu capture at 64
# experts and 512 tokens (one chunk per expert, as in the full workload) scaled by the full
# workload's 4x weight bytes and pairs.
TC_GATE_UP_TRAFFIC = 4 * (580347392 + 58900992)
# The same for one expert_ffn_kernel launch (the 4096 -> 2048 -> 4096 expert, one launch).
EXPERT_FFN_TRAFFIC = 12829440 + 0


def max_over_ranks(t, world, device):
    """The job's time: the largest of the ranks' times (the job ends with its
    slowest replica). All ranks must call it when world > 1."""
    if world <= 1:
        return t
    import torch
    import torch.distributed as dist
    tt = torch.tensor([float(t)], device=device, dtype=torch.float64)
    dist.all_reduce(tt, op=dist.ReduceOp.MAX)
    return float(tt.item())


def job_rate(units_per_rank, world, t):
    """Whole-job throughput: the units all ranks processed over the job's time."""
    return units_per_rank * world / t


def _tensor_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["bf16_tflops_sustained"]), "measured (MEASURED_PEAKS.json bf16_tflops_sustained)"
    except Exception:
        return 1700.0, "fallback 1.7 PFLOP/s sustained"


def bytes_per_token(layer=None):
    """(bytes one token reads: the selected experts' blocks and the router;
    gate/up bytes; down bytes), tq2_0_fx4 unless a layer says otherwise."""
    from paper_2608_08910_gb300 import binding as B
    mg = layer.mb_gu if layer is not None else B.tqfx4_matrix_bytes(I, H)
    md = layer.mb_d if layer is not None else B.tqfx4_matrix_bytes(H, I)
    return TOPK * (2 * mg + md) + E * H * 4, TOPK * 2 * mg, TOPK * md


class ClockSampler:
    """nvidia-smi clock and throttle-reason samples while the timed region runs."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.samples = []
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.QUERY, "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.samples.append([x.strip() for x in line.split(",")])

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.2)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        sm = [float(s[1]) for s in self.samples if s[1].replace(".", "", 1).isdigit()]
        mx = [float(s[2]) for s in self.samples if s[2].replace(".", "", 1).isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = set()
        for s in self.samples:
            for n, v in zip(names, s[5:9]):
                if v.strip().lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(self.samples)}


def cpu_baseline(seconds_budget=20.0, tokens=None, layer=None):
    """The oracle (plain single-threaded C) on a bounded sample of the same
    workload: whole tokens through the MoE layer, packing of the experts they
    select excluded from the time (layer: an MXFP4 layer whose expert bytes
    the oracle reads instead). Returns (GB/s, tokens, seconds)."""
    import numpy as np
    import torch

    import oracle
    from paper_2608_08910_gb300 import inputs

    dev = "cuda" if torch.cuda.is_available() else "cpu"
    Wr = inputs.router_weight(SEED, E, H, dev).cpu().numpy()
    X = inputs.hidden_states(SEED, POOL, H, dev).cpu().numpy()
    per_token, _, _ = bytes_per_token(layer)
    total_t, done = 0.0, 0
    n_max = tokens if tokens else POOL
    for t in range(n_max):
        _, idx, _ = oracle.router(Wr, None, X[t], TOPK)
        if layer is not None:
            ex = {int(e): tuple(b.cpu().numpy() for b in layer.expert_blocks(int(e))) for e in idx}
        else:
            ex = {int(e): tuple(oracle.pack_rtn(inputs.expert_matrix(SEED, int(e), p, H, I, dev).cpu().numpy())
                                for p in (0, 1, 2)) for e in idx}
        t0 = time.perf_counter()
        oracle.moe_tokens(ex, E, H, I, Wr, None, TOPK, X[t], fmt="mxfp4" if layer is not None else "fx4")
        total_t += time.perf_counter() - t0
        done += 1
        if tokens is None and total_t >= seconds_budget:
            break
    return per_token * done / total_t / 1e9, done, total_t


def cpu_baseline_all_cores(tokens_per_core=2):
    """The same oracle on all host cores: one Python thread per core, each
    running whole tokens through the MoE layer (the oracle's C calls release
    the interpreter lock, so the threads run in parallel). The experts of
    the sampled tokens are packed first, outside the timed region. Returns
    (GB/s, tokens, seconds, threads)."""
    import concurrent.futures

    import torch

    import oracle
    from paper_2608_08910_gb300 import inputs

    cores = os.cpu_count() or 1
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    Wr = inputs.router_weight(SEED, E, H, dev).cpu().numpy()
    X = inputs.hidden_states(SEED, POOL, H, dev).cpu().numpy()
    n_tok = min(POOL, cores * tokens_per_core)
    per_token, _, _ = bytes_per_token()
    ex = {}
    for t in range(n_tok):
        _, idx, _ = oracle.router(Wr, None, X[t], TOPK)
        for e in idx:
            if int(e) not in ex:
                ex[int(e)] = tuple(oracle.pack_rtn(inputs.expert_matrix(SEED, int(e), p, H, I, dev).cpu().numpy())
                                   for p in (0, 1, 2))

    def work(t):
        oracle.moe_tokens(ex, E, H, I, Wr, None, TOPK, X[t])

    with concurrent.futures.ThreadPoolExecutor(max_workers=cores) as pool:
        t0 = time.perf_counter()
        list(pool.map(work, range(n_tok)))
        el = time.perf_counter() - t0
    return per_token * n_tok / el / 1e9, n_tok, el, cores


def run_reference(args, rank, world):
    """--impl reference: the CPU oracle, as it stands, on this machine's host
    cores; each step is one expert FFN of a routed token (1/8 of a token)."""
    if rank != 0:
        return
    import numpy as np
    import torch

    import oracle
    from paper_2608_08910_gb300 import binding as B
    from paper_2608_08910_gb300 import inputs

    dev = "cuda" if torch.cuda.is_available() else "cpu"
    Wr = inputs.router_weight(SEED, E, H, dev).cpu().numpy()
    X = inputs.hidden_states(SEED, POOL, H, dev).cpu().numpy()
    mb = B.tqfx4_matrix_bytes(I, H)
    cache = {}

    def expert(e):
        if e not in cache:
            cache.clear()
            cache[e] = tuple(oracle.pack_rtn(inputs.expert_matrix(SEED, e, p, H, I, dev).cpu().numpy())
                             for p in (0, 1, 2))
        return cache[e]

    def step(s):
        t = s // TOPK
        _, idx, _ = oracle.router(Wr, None, X[t % POOL], TOPK)
        g, u, d = expert(int(idx[s % TOPK]))
        t0 = time.perf_counter()
        oracle.expert_ffn(g, u, d, H, I, X[t % POOL])
        return time.perf_counter() - t0

    for s in range(args.warmup):
        step(s)
    el = sum(step(args.warmup + s) for s in range(args.steps))
    bytes_step = 3 * mb
    value = bytes_step * args.steps / el / 1e9
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": el / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "i8xi4-i32,f32",
        "data": "synthetic", "config": {"workload": WORKLOAD, "sample": "one expert FFN per step (1/8 token)"},
        "cpu_baseline": {"value": value, "unit": "GB/s", "cores": 1, "kind": "oracle",
                         "sample": "%d expert FFNs of routed tokens, packing excluded" % args.steps},
        "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_grouped(args, rank, world, local):
    """Batched decode (64 tokens, Zipf(1.1) router bias) or prefill (2048
    tokens) through tqfx4_moe_grouped; one step = one call over the batch.
    Metric: tokens/s, with the effective GB/s of the touched experts' blocks
    and, for prefill, the dense-equivalent TFLOP/s of the expert GEMMs."""
    import torch
    import torch.distributed as dist

    from paper_2608_08910_gb300 import binding as B
    from paper_2608_08910_gb300 import inputs
    from paper_2608_08910_gb300.moe import MoeLayer

    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    T, zipf, path = (64, 1.1, B.TQFX4_PATH_AUTO) if args.workload == "grouped_decode_64" else \
        (2048, 0.0, B.TQFX4_PATH_PREFILL)
    if args.tokens:
        T = args.tokens
    dev = torch.device("cuda", local)
    layer = MoeLayer.synthetic(SEED, E, H, I, TOPK, zipf, dev)
    ws = layer.workspace(T, path)
    n_batches = 4
    Xs = [inputs.hidden_states(SEED + 97 * b + rank, T, H, dev) for b in range(n_batches)]
    OUT = torch.empty((T, H), device=dev)
    sel = torch.empty((T, TOPK), dtype=torch.int32, device=dev)
    selw = torch.empty((T, TOPK), device=dev)
    stream = torch.cuda.current_stream(dev)
    for i in range(args.warmup):
        layer.grouped(Xs[i % n_batches], ws, path, OUT, sel, selw, stream=stream)
    B.tqfx4_check(ws)
    mb = B.tqfx4_matrix_bytes(I, H)
    touched = 0
    hits = None  # (token, slot) pairs per expert of the first batch, descending
    for X in Xs:
        layer.grouped(X, ws, path, OUT, sel, selw, stream=stream)
        counts = torch.bincount(sel.flatten().long(), minlength=E)
        touched += int((counts > 0).sum())
        if hits is None:
            hits = sorted(counts.tolist(), reverse=True)
    bytes_per_step = touched / n_batches * 3 * mb + E * H * 4
    # The K steps are captured once into a CUDA graph (as a serving loop
    # would run them), so the timed region holds no host launch work.
    cap_stream = torch.cuda.Stream(dev)
    cap_stream.wait_stream(stream)
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(cap_stream):
        with torch.cuda.graph(graph, stream=cap_stream):
            for i in range(args.steps):
                layer.grouped(Xs[i % n_batches], ws, path, OUT, sel, selw, stream=cap_stream)
    stream.wait_stream(cap_stream)
    graph.replay()  # untimed
    torch.cuda.synchronize()
    B.tqfx4_check(ws)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clk:
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        ev0.record(stream)
        graph.replay()
        ev1.record(stream)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
    B.tqfx4_check(ws)
    t = ev0.elapsed_time(ev1) / 1e3
    t = max_over_ranks(t, world, dev)
    tokens = T * args.steps * world  # tokens of the whole job
    # per-stage device times (CUDA events on the launching stream)
    n_st = B.tqfx4_moe_stage_count(1, path)
    names = [B.tqfx4_moe_stage_name(1, path, s) for s in range(n_st)]
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(n_st + 1)]
    for e_ in evs:
        e_.record(stream)
    acc = [0.0] * n_st
    reps = min(args.steps, 10)
    for i in range(reps):
        layer.grouped(Xs[i % n_batches], ws, path, OUT, sel, selw, stream=stream, events=evs)
        evs[-1].synchronize()
        for s in range(n_st):
            acc[s] += evs[s].elapsed_time(evs[s + 1]) / 1e3
    stage_s = {names[s]: acc[s] / reps for s in range(n_st)}
    peak_hbm, peak_kind = _peaks()
    flops_gu = 2.0 * T * TOPK * 2 * I * H
    # end to end through the public API's host-buffer call
    # (tqfx4_moe_grouped_host): the batch's hidden states from pinned host
    # memory, the outputs and expert ids into it, every step
    Xh = [x.cpu().pin_memory() for x in Xs]
    outh = torch.empty((T, H), pin_memory=True)
    selh = torch.empty((T, TOPK), dtype=torch.int32, pin_memory=True)
    ws_h = layer.grouped_host_workspace(T, path)
    for i in range(2):
        layer.grouped_host(Xh[i % n_batches], ws_h, outh, selh, None, path, stream=stream)
    torch.cuda.synchronize()
    ev0.record(stream)
    for i in range(args.steps):
        layer.grouped_host(Xh[i % n_batches], ws_h, outh, selh, None, path, stream=stream)
    ev1.record(stream)
    torch.cuda.synchronize()
    B.tqfx4_check(ws_h)
    te = ev0.elapsed_time(ev1) / 1e3
    te = max_over_ranks(te, world, dev)
    if path == B.TQFX4_PATH_PREFILL:
        # the dominant kernel is the tensor-core contraction of gate and up:
        # dense-equivalent flops over its time, against the measured bf16 peak
        peak_tc, tc_kind = _tensor_peak()
        achieved = flops_gu / stage_s["gate_up"] / 1e12
        roof = {"bound": "tensor", "achieved": achieved, "peak": peak_tc, "unit": "TFLOP/s",
                "frac": achieved / peak_tc,
                "kernel": "gate_up stage: tc_gemm_kernel, then small_groups_kernel (chunks of <= 4 pairs, if any)",
                "traffic": TC_GATE_UP_TRAFFIC if (T == 2048 and E == 256) else None,
                "traffic_source": "ncu capture at 64 experts / 512 tokens, scaled x4",
                "peak_source": tc_kind}
    else:
        gu_bytes = touched / n_batches * 2 * mb
        achieved = gu_bytes / stage_s["gate_up"] / 1e9
        roof = {"bound": "hbm", "achieved": achieved, "peak": peak_hbm, "unit": "GB/s",
                "frac": achieved / peak_hbm, "traffic": None,
                "kernel": "gate_up stage: tc_gemm_kernel (chunks of > 4 pairs), then small_groups_kernel",
                "peak_source": peak_kind}
    roof["stage_us"] = {k: v * 1e6 for k, v in stage_s.items()}
    line = {
        "metric": "MoE-layer tokens/s (%s)" % args.workload, "value": job_rate(T * args.steps, world, t),
        "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": t / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "i8xi4-i32,f32",
        "data": "synthetic",
        "config": {"workload": args.workload, "tokens": T, "experts": E, "hidden": H, "inter": I, "top_k": TOPK,
                   "zipf": zipf, "touched_experts_avg": touched / n_batches, "seed": SEED,
                   "expert_hits_first_batch": {"top16": hits[:16], "experts_with_1": hits.count(1),
                                               "experts_with_2_to_4": sum(1 for h in hits if 2 <= h <= 4),
                                               "touched": sum(1 for h in hits if h > 0)},
                   "l2": "inputs larger than L2 (3.27 GB expert pool); 4 batches cycled"},
        "effective_gbs": bytes_per_step * args.steps * world / t / 1e9,
        "roofline": roof,
        "e2e": {"value": tokens / te, "unit": "tokens/s", "h2d_bytes_per_step": T * H * 4,
                "d2h_bytes_per_step": T * H * 4 + T * TOPK * 4},
        # router (norms, screening GEMM and refinement from 256 tokens, else one kernel), top-k, group,
        # quantize, activation planes, gather, gate/up (tensor cores, then the small-group pass), SwiGLU,
        # down (the same two), combine
        "gpu_launches": ((3 if T >= 256 else 1) + 11) * args.steps,
        "clocks": clk.summary(),
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def run_tiered(args, rank, world, local):
    """One token per step through the 256-expert layer with every expert in
    pinned host memory and a device slab of --slots experts (the expert tier):
    route on the GPU, read the selection on the host, copy each missing
    expert's blocks into a slot (one contiguous range per projection), then
    the expert projections. Uniform routing over 256 experts with 8 slots
    misses on almost every lookup, so this is the miss-bound rate of the
    paper's streamed store, with the host link in the place of its SSD. The
    host reads the selection every token, so the steps are not graph-captured."""
    import torch
    import torch.distributed as dist

    from paper_2608_08910_gb300 import binding as B
    from paper_2608_08910_gb300 import inputs
    from paper_2608_08910_gb300.moe import MoeLayer
    from paper_2608_08910_gb300.tier import ExpertTier

    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    assert args.warmup >= 3, "at least 3 warm-up steps"
    dev = torch.device("cuda", local)
    layer = MoeLayer.synthetic(SEED, E, H, I, TOPK, 0.0, dev)
    tier = ExpertTier(layer, args.slots)
    ws = layer.workspace(1)
    X = inputs.hidden_states(SEED + rank, POOL, H, dev)
    Xh = X.cpu().pin_memory()
    xin = torch.empty(H, device=dev)
    out = torch.empty(H, device=dev)
    outh = torch.empty(H, pin_memory=True)
    sel = torch.empty(TOPK, dtype=torch.int32, device=dev)
    selw = torch.empty(TOPK, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step(i):
        xin.copy_(Xh[i % POOL], non_blocking=True)
        tier.ffn(xin, ws, out, sel, selw, stream)
        outh.copy_(out, non_blocking=True)

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    B.tqfx4_check(ws)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def timed(first):
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        ev0.record(stream)
        for i in range(args.steps):
            step(first + i)
        ev1.record(stream)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        return ev0.elapsed_time(ev1) / 1e3

    # The host waits for the selection every token, and nvidia-smi queries
    # stall such host-synchronous loops (measured: a quarter of the rate), so
    # the clocks are sampled over an adjacent run of the same steps and the
    # reported time is the run without the sampler.
    with ClockSampler(local) as clk:
        t_sampled = timed(args.warmup)
    m0, l0 = tier.misses, tier.lookups
    t = max_over_ranks(timed(args.warmup + args.steps), world, dev)
    B.tqfx4_check(ws)
    misses, lookups = tier.misses - m0, tier.lookups - l0
    expert_bytes = 2 * layer.mb_gu + layer.mb_d
    miss_bytes = misses * expert_bytes
    # the link's copy rate: one pinned host -> device copy of top_k experts'
    # bytes (a token's misses), timed alone
    probe_h = tier.host[:TOPK].reshape(-1)  # top_k experts' bytes
    probe_d = torch.empty_like(probe_h, device=dev)
    for _ in range(3):
        probe_d.copy_(probe_h, non_blocking=True)
    torch.cuda.synchronize()
    ev0.record(stream)
    for _ in range(10):
        probe_d.copy_(probe_h, non_blocking=True)
    ev1.record(stream)
    torch.cuda.synchronize()
    link_gbs = 10 * probe_h.numel() / (ev0.elapsed_time(ev1) / 1e3) / 1e9
    achieved = miss_bytes / t / 1e9
    line = {
        "metric": "MoE-layer tokens/s, experts in host memory (tiered_decode)",
        "value": job_rate(args.steps, world, t), "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": t / args.steps * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "i8xi4-i32,f32", "data": "synthetic",
        "config": {"workload": "tiered_decode", "experts": E, "hidden": H, "inter": I, "top_k": TOPK,
                   "slots": args.slots, "routing": "uniform", "tokens_per_step": 1,
                   "l2": "experts streamed from host memory; 3.27 GB pool"},
        "miss_rate": misses / max(1, lookups),
        "roofline": {"bound": "host-link", "achieved": achieved, "peak": link_gbs, "unit": "GB/s",
                     "frac": achieved / link_gbs, "traffic": None, "kernel": "expert misses (cudaMemcpyAsync)",
                     "peak_source": "measured in this run: pinned host -> device copy of %d bytes" % probe_h.numel()},
        "e2e": {"value": job_rate(args.steps, world, t), "unit": "tokens/s", "h2d_bytes_per_step": H * 4,
                "d2h_bytes_per_step": H * 4 + TOPK * 4},
        "gpu_launches": 3 * args.steps,
        "clocks": dict(clk.summary(), note="sampled over an adjacent run of the same steps (%.3f ms per step "
                                           "with the sampler running)" % (t_sampled / args.steps * 1e3)),
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()

GEMV_N, GEMV_K, GEMV_POOL = 131072, 4096, 16
# DRAM bytes (read + write) of one launch of the GEMV kernels on the 131072 x
# 4096 workload, from ncu --set full captures (profiles/); None once a kernel
# changes until it is captured again.
GEMV_TRAFFIC = {"mxfp4_gemv": 285286144 + 3272960, "free_gemv": 276858112 + 3605504}


def run_gemv(args, rank, world, local):
    """One GEMV per step over a 131072 x 4096 matrix (64 experts' 2048 x 4096
    gate projections stacked, larger than L2) in a second weight format, a new
    activation every step: tqfx4_quantize_act, then the format's dot pass.
    mxfp4_gemv: MXFP4 blocks (the released bytes, 17 per 32 elements, 285 MB)
    through tqfx4_gemv_mxfp4; free_gemv: the free-scale two-plane blocks
    (528 bytes per 4 x 256, 277 MB) through tqfx4_gemv_free. The tq2_0_fx4
    GEMV of a matrix of the same shape is timed beside it (for free_gemv this
    is the paper's fold-versus-planes speed ablation). Metric: effective GB/s
    of the format's bytes over the step time."""
    import torch
    import torch.distributed as dist

    from paper_2608_08910_gb300 import binding as B
    from paper_2608_08910_gb300 import inputs, ops

    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    assert args.warmup >= 3, "at least 3 warm-up steps"
    dev = torch.device("cuda", local)
    n, k = GEMV_N, GEMV_K
    ws = ops.workspace(B.TQFX4_STATUS_BYTES, dev)
    free = args.workload == "free_gemv"
    if free:
        t1, t2, s1 = inputs.trit_planes(SEED, n, k, dev)
        s2 = inputs.trit_planes(SEED + 1, n, k, dev)[2]
        mx = ops.pack_free(t1, t2, s1.view(torch.int16), s2.view(torch.int16), ws)
        del t1, t2
    else:
        mx = inputs.mxfp4_matrix(SEED, n, k, dev)
    mx_bytes = mx.numel()
    fx = ops.pack_rtn(inputs.gemv_matrix(SEED, n, k, dev), ws)
    fx_bytes = fx.numel()
    torch.cuda.empty_cache()
    X = inputs.hidden_states(SEED + rank, GEMV_POOL, k, dev)
    q = torch.empty(k, dtype=torch.int8, device=dev)
    da = torch.empty(k // 256, device=dev)
    bs = torch.empty(k // 256, dtype=torch.int32, device=dev)
    y = torch.empty(n, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step(i, fmt="mxfp4", st=stream, ev=None):
        if ev:
            ev[0].record(st)
        B.tqfx4_quantize_act(X[i % GEMV_POOL], 1, k, q, da, bs, ws, st)
        if ev:
            ev[1].record(st)
        if fmt == "mxfp4":
            B.tqfx4_gemv_mxfp4(mx, n, k, q, da, y, None, ws, st)
        elif fmt == "free":
            B.tqfx4_gemv_free(mx, n, k, q, da, bs, y, None, None, ws, st)
        else:
            B.tqfx4_gemv(fx, n, k, q, da, bs, y, None, ws, st)
        if ev:
            ev[2].record(st)

    def graph_of(fmt):
        for i in range(args.warmup):
            step(i, fmt)
        torch.cuda.synchronize()
        B.tqfx4_check(ws)
        cap = torch.cuda.Stream(dev)
        cap.wait_stream(stream)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.stream(cap):
            with torch.cuda.graph(g, stream=cap):
                for i in range(args.steps):
                    step(args.warmup + i, fmt, st=cap)
        stream.wait_stream(cap)
        g.replay()  # untimed
        torch.cuda.synchronize()
        return g

    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def timed(g):
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        ev0.record(stream)
        g.replay()
        ev1.record(stream)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        return max_over_ranks(ev0.elapsed_time(ev1) / 1e3, world, dev)

    fmt = "free" if free else "mxfp4"
    g_mx = graph_of(fmt)
    with ClockSampler(local) as clk:
        t = timed(g_mx)
    B.tqfx4_check(ws)
    t_fx = timed(graph_of("fx4"))
    B.tqfx4_check(ws)

    def stage_times(fmt):
        reps = min(args.steps, 20)
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(reps)]
        for i in range(reps):
            step(i, fmt, ev=evs[i])
        torch.cuda.synchronize()
        return (sum(e[0].elapsed_time(e[1]) for e in evs) / reps / 1e3,
                sum(e[1].elapsed_time(e[2]) for e in evs) / reps / 1e3)

    q_mx, g_mx_s = stage_times(fmt)
    _, g_fx_s = stage_times("fx4")
    B.tqfx4_check(ws)

    # end to end: the activation from pinned host memory, y back to it
    Xh = X.cpu().pin_memory()
    xin = torch.empty(k, device=dev)
    yh = torch.empty(n, pin_memory=True)

    def step_e2e():
        B.tqfx4_quantize_act(xin, 1, k, q, da, bs, ws, stream)
        if free:
            B.tqfx4_gemv_free(mx, n, k, q, da, bs, y, None, None, ws, stream)
        else:
            B.tqfx4_gemv_mxfp4(mx, n, k, q, da, y, None, ws, stream)
        yh.copy_(y, non_blocking=True)

    for i in range(3):
        xin.copy_(Xh[i], non_blocking=True)
        step_e2e()
    torch.cuda.synchronize()
    ev0.record(stream)
    for i in range(args.steps):
        xin.copy_(Xh[i % GEMV_POOL], non_blocking=True)
        step_e2e()
    ev1.record(stream)
    torch.cuda.synchronize()
    B.tqfx4_check(ws)
    te = max_over_ranks(ev0.elapsed_time(ev1) / 1e3, world, dev)

    peak, peak_kind = _peaks()
    achieved = mx_bytes / g_mx_s / 1e9
    line = {
        "metric": ("effective free-scale two-plane GB/s (GEMV, 131072 x 4096)" if free
                   else "effective MXFP4 GB/s (GEMV, 131072 x 4096)"),
        "value": job_rate(mx_bytes * args.steps, world, t) / 1e9, "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": t / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "i8xi2-i32,f32" if free else "i8xe2m1-i32,f32", "data": "synthetic",
        "config": {"workload": args.workload, "n": n, "k": k, "matrix_bytes": mx_bytes,
                   "l2": "inputs larger than L2 (%d MB matrix); a different activation per step" % (mx_bytes >> 20)},
        "fx4_same_shape": {"gbs": fx_bytes * args.steps / t_fx / 1e9, "ms_per_step": t_fx / args.steps * 1e3,
                           "matrix_bytes": fx_bytes, "gemv_us": g_fx_s * 1e6,
                           "gemv_gbs": fx_bytes / g_fx_s / 1e9},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": GEMV_TRAFFIC[args.workload],
                     "kernel": "gemv_free_kernel" if free else "mxfp4_gemv_kernel",
                     "peak_source": peak_kind, "stage_us": {"quantize_act": q_mx * 1e6, "gemv": g_mx_s * 1e6}},
        "e2e": {"value": job_rate(mx_bytes * args.steps, world, te) / 1e9, "unit": "GB/s",
                "h2d_bytes_per_step": k * 4, "d2h_bytes_per_step": n * 4},
        "gpu_launches": 2 * args.steps,
        "clocks": clk.summary(),
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import numpy as np

        import oracle
        rows = 2048
        sub = mx[:rows * (mx_bytes // n)].cpu().numpy()
        qh, dah = q.cpu().numpy(), da.cpu().numpy()
        done, el = 0, 0.0
        while el < 10.0:
            t0 = time.perf_counter()
            (oracle.free_gemv if free else oracle.mxfp4_gemv)(sub, rows, k, qh, dah)
            el += time.perf_counter() - t0
            done += 1
        line["cpu_baseline"] = {"value": done * sub.nbytes / el / 1e9, "unit": "GB/s", "cores": 1,
                                "kind": "oracle", "sample": "%d GEMVs of the matrix's first %d rows" % (done, rows)}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


SMALL_POOL_BYTES = 256 << 20  # distinct weight bytes rotated through the steps of gemv_1024 / expert_ffn


def run_small(args, rank, world, local):
    """The two single-matrix workloads, each on a pool of distinct weights
    larger than L2 (at least 256 MB), one pool entry per step, a new
    activation every step:
    gemv_1024: one 1024 x 1024 tq2_0_fx4 GEMV (round-to-nearest codes of
      N(0, 0.02) weights) of an N(0, 1) vector quantized per block:
      tqfx4_gemv_x (the quantization and the GEMV in one launch); 505
      matrices (269 MB) rotated.
    expert_ffn: one SwiGLU expert, gate/up 4096 -> 2048, down 2048 -> 4096,
      Student-t(5) x 0.02 weights: tqfx4_expert_ffn (the expert alone, no
      router: one cooperative launch that holds the expert on chip, with
      the quantization of x inside); 21 such experts (268 MB) rotated.
    Metric: effective GB/s of the matrices' blocks over the step time. The
    same steps on one resident matrix (hot L2) are reported beside it."""
    import torch
    import torch.distributed as dist

    from paper_2608_08910_gb300 import binding as B
    from paper_2608_08910_gb300 import inputs, ops
    from paper_2608_08910_gb300.moe import MoeLayer

    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    assert args.warmup >= 3, "at least 3 warm-up steps"
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream(dev)
    gemv = args.workload == "gemv_1024"
    xpool = 64
    if gemv:
        n = k = 1024
        mat = B.tqfx4_matrix_bytes(n, k)
        M = (SMALL_POOL_BYTES + mat - 1) // mat
        ws = ops.workspace(B.TQFX4_STATUS_BYTES, dev)
        # M matrices stacked as one (M n) x k matrix: matrix i is row groups [i n/4, (i+1) n/4)
        pool = ops.pack_rtn(inputs.gemv_matrix(SEED, M * n, k, dev), ws)
        torch.cuda.empty_cache()
        X = inputs.hidden_states(SEED + rank, xpool, k, dev)
        y = torch.empty(n, device=dev)
        step_bytes = mat

        def step(i, st=stream, hot=False, ev=None, x=None):
            if ev:
                ev[0].record(st)
            m = 0 if hot else i % M
            B.tqfx4_gemv_x(pool[m * mat:(m + 1) * mat], n, k, X[i % xpool] if x is None else x, y, None, None,
                           None, ws, st)
            if ev:
                ev[1].record(st)
        launches = 1
        kern = "gemv_chunk_kernel (quantization inside)"
        cfg = {"workload": "gemv_1024x1024", "n": n, "k": k, "matrix_bytes": mat, "pool_matrices": M,
               "l2": "inputs larger than L2: %d distinct matrices (%d MB) rotated, a new activation per step"
                     % (M, M * mat >> 20)}
    else:
        Hh, Ii = H, I
        mat = 2 * B.tqfx4_matrix_bytes(Ii, Hh) + B.tqfx4_matrix_bytes(Hh, Ii)
        M = (SMALL_POOL_BYTES + mat - 1) // mat
        layers = [MoeLayer.synthetic(SEED + m, 1, Hh, Ii, 1, 0.0, dev) for m in range(M)]
        torch.cuda.empty_cache()
        ws = layers[0].expert_workspace()
        X = inputs.hidden_states(SEED + rank, xpool, Hh, dev)
        out = torch.empty(Hh, device=dev)
        step_bytes = mat

        def step(i, st=stream, hot=False, ev=None, x=None):
            L = layers[0 if hot else i % M]
            L.expert_ffn(0, X[i % xpool] if x is None else x, ws, out, stream=st, events=ev)
        launches = B.tqfx4_expert_ffn_launches(Hh, Ii)
        kern = "expert_ffn_kernel (one cooperative launch)" if launches == 1 else "gate_up"
        cfg = {"workload": "expert_ffn_h4096_i2048", "hidden": Hh, "inter": Ii, "expert_bytes": mat,
               "pool_experts": M, "call": "tqfx4_expert_ffn (no router)",
               "l2": "inputs larger than L2: %d distinct experts (%d MB) rotated, a new activation per step"
                     % (M, M * mat >> 20)}

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    B.tqfx4_check(ws)

    def graph_of(hot):
        cap = torch.cuda.Stream(dev)
        cap.wait_stream(stream)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.stream(cap):
            with torch.cuda.graph(g, stream=cap):
                for i in range(args.steps):
                    step(args.warmup + i, st=cap, hot=hot)
        stream.wait_stream(cap)
        g.replay()  # untimed
        torch.cuda.synchronize()
        return g

    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def timed(g):
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        ev0.record(stream)
        g.replay()
        ev1.record(stream)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        return max_over_ranks(ev0.elapsed_time(ev1) / 1e3, world, dev)

    g_cold = graph_of(False)
    with ClockSampler(local) as clk:
        t = timed(g_cold)
    B.tqfx4_check(ws)
    reps = [timed(g_cold) for _ in range(3)]
    t_hot = timed(graph_of(True))
    B.tqfx4_check(ws)

    # the dominant kernel's duration: CUDA events around each stage of every
    # step, on the launching stream, in plain stream order (the library's
    # traced call records its own stage events; the GEMV steps are not
    # captured, since an event recorded by torch inside a capture does not time)
    n_ev = 2 if gemv else 3  # the traced expert call records three events either way
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(n_ev)] for _ in range(args.steps)]
    for row in evs:
        for e_ in row:
            e_.record(stream)
    torch.cuda.synchronize()
    if gemv:
        for i in range(args.steps):
            step(args.warmup + i, ev=evs[i])
    else:
        cap = torch.cuda.Stream(dev)
        cap.wait_stream(stream)
        g_ev = torch.cuda.CUDAGraph()
        with torch.cuda.stream(cap):
            with torch.cuda.graph(g_ev, stream=cap):
                for i in range(args.steps):
                    step(args.warmup + i, st=cap, ev=evs[i])
        stream.wait_stream(cap)
        g_ev.replay()
    torch.cuda.synchronize()
    B.tqfx4_check(ws)
    stage = [sum(r[s].elapsed_time(r[s + 1]) for r in evs) / args.steps / 1e3 for s in range(n_ev - 1)]
    if gemv:
        names = ["gemv_x"]
        dom_s, dom_bytes = stage[0], mat
    elif launches == 1:
        names = ["expert_ffn"]
        dom_s, dom_bytes = stage[0], mat
    else:
        names = ["gate_up", "down"]
        dom_s, dom_bytes = stage[0], 2 * B.tqfx4_matrix_bytes(I, H)
    stage_us = {names[s]: stage[s] * 1e6 for s in range(len(names))}

    # end to end through the public API's host-buffer calls (tqfx4_gemv_x_host,
    # tqfx4_expert_ffn_host): x from pinned host memory, y (out) into it, every
    # step; plain calls, no graph
    xrows = [r for r in X.cpu().pin_memory()]
    resh = torch.empty(n if gemv else Hh, pin_memory=True)
    if gemv:
        ws_h = ops.gemv_x_host_workspace(n, k, dev)

        def step_h(i):
            m = i % M
            ops.gemv_x_host(pool[m * mat:(m + 1) * mat], n, k, xrows[i % xpool], resh, ws_h, stream)
    else:
        ws_h = layers[0].expert_host_workspace()

        def step_h(i):
            layers[i % M].expert_ffn_host(0, xrows[i % xpool], ws_h, resh, stream=stream)
    for i in range(3):
        step_h(i)
    torch.cuda.synchronize()
    ev0.record(stream)
    for i in range(args.steps):
        step_h(args.warmup + i)
    ev1.record(stream)
    torch.cuda.synchronize()
    B.tqfx4_check(ws_h)
    te = max_over_ranks(ev0.elapsed_time(ev1) / 1e3, world, dev)

    peak, peak_kind = _peaks()
    achieved = dom_bytes / dom_s / 1e9
    line = {
        "metric": "effective tq2_0_fx4 GB/s (%s)" % ("GEMV 1024 x 1024" if gemv else "one expert SwiGLU FFN"),
        "value": job_rate(step_bytes * args.steps, world, t) / 1e9, "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": t / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "i8xi4-i32,f32",
        "data": "synthetic", "config": cfg,
        "steps_per_s": job_rate(args.steps, world, t),
        "repeats_ms_per_step": [r / args.steps * 1e3 for r in reps],
        "hot_l2": {"value": step_bytes * args.steps / t_hot / 1e9, "unit": "GB/s",
                   "ms_per_step": t_hot / args.steps * 1e3,
                   "note": "the same steps on one resident matrix (L2-resident after the first step)"},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                     "traffic": EXPERT_FFN_TRAFFIC if (not gemv and launches == 1) else None, "kernel": kern,
                     "peak_source": peak_kind + " (MEASURED_PEAKS.json hbm_gbs)" if peak_kind == "measured"
                     else "fallback 6.8 TB/s",
                     "stage_us": stage_us,
                     "note": ("a single-wave launch of 32 CTAs: bound by latency (launch, one copy round trip), "
                              "not by HBM" if gemv else
                              "all three matrices of the expert in one launch: bound by the chain of copy, "
                              "grid barrier and the two dot passes, not by HBM" if launches == 1
                              else "the gate and up projections of one expert")},
        "e2e": {"value": job_rate(step_bytes * args.steps, world, te) / 1e9, "unit": "GB/s",
                "h2d_bytes_per_step": X.shape[1] * 4, "d2h_bytes_per_step": resh.numel() * 4},
        "gpu_launches": launches * args.steps,
        "clocks": clk.summary(),
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import concurrent.futures

        import numpy as np

        import oracle
        xs = X[:8].cpu().numpy()
        if gemv:
            blocks = oracle.pack_rtn(inputs.gemv_matrix(SEED, n, k).numpy())

            def one(i):
                rq, rda, _ = oracle.quantize_act(xs[i % 8])
                oracle.gemv(blocks, n, k, rq, rda)
        else:
            ex = tuple(oracle.pack_rtn(inputs.expert_matrix(SEED, 0, p, H, I, dev).cpu().numpy()) for p in (0, 1, 2))

            def one(i):
                oracle.expert_ffn(*ex, H, I, xs[i % 8])
        done, el = 0, 0.0
        while el < 10.0:
            t0 = time.perf_counter()
            one(done)
            el += time.perf_counter() - t0
            done += 1
        line["cpu_baseline"] = {"value": done * step_bytes / el / 1e9, "unit": "GB/s", "cores": 1, "kind": "oracle",
                                "sample": "%d %s on one core (%.1f s)" % (done, "GEMVs" if gemv else "expert FFNs", el)}
        cores = os.cpu_count() or 1
        n_all = done * cores // 2 if gemv else 2 * cores
        with concurrent.futures.ThreadPoolExecutor(max_workers=cores) as ex_:
            t0 = time.perf_counter()
            list(ex_.map(one, range(n_all)))
            el_all = time.perf_counter() - t0
        line["cpu_baseline_all_cores"] = {"value": n_all * step_bytes / el_all / 1e9, "unit": "GB/s", "cores": cores,
                                          "kind": "oracle", "sample": "%d steps on %d threads (%.1f s wall)"
                                          % (n_all, cores, el_all)}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


PACK_MATS = 8  # distinct 2048 x 4096 fp32 expert matrices cycled (268 MB, larger than L2)


def run_pack(args, rank, world, local):
    """The tied alternating solver (Sec. 2.1) as a pack source: one step packs
    one 2048 x 4096 fp32 expert projection (Student-t(5) x 0.02) into
    tq2_0_fx4 blocks through tqfx4_pack(TQFX4_SRC_F32_TIED); eight matrices
    are cycled. Round-to-nearest packing of the same matrices is timed
    beside it. Metric: expert matrices packed per second."""
    import torch
    import torch.distributed as dist

    from paper_2608_08910_gb300 import binding as B
    from paper_2608_08910_gb300 import inputs, ops

    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    assert args.warmup >= 3, "at least 3 warm-up steps"
    dev = torch.device("cuda", local)
    n, k = I, H  # a gate projection: 2048 x 4096
    W = [inputs.expert_matrix(SEED, e, inputs.PROJ_GATE, H, I, dev) for e in range(PACK_MATS)]
    ws = ops.workspace(B.TQFX4_STATUS_BYTES, dev)
    out = ops.empty_blocks(n, k, dev)
    stream = torch.cuda.current_stream(dev)

    def step(i, src=B.TQFX4_SRC_F32_TIED, st=stream):
        B.tqfx4_pack(src, W[i % PACK_MATS], None, None, n, k, out, ws, st)

    def graph_of(src):
        for i in range(args.warmup):
            step(i, src)
        torch.cuda.synchronize()
        B.tqfx4_check(ws)
        cap = torch.cuda.Stream(dev)
        cap.wait_stream(stream)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.stream(cap):
            with torch.cuda.graph(g, stream=cap):
                for i in range(args.steps):
                    step(i, src, st=cap)
        stream.wait_stream(cap)
        g.replay()
        torch.cuda.synchronize()
        return g

    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def timed(g):
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        ev0.record(stream)
        g.replay()
        ev1.record(stream)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        return max_over_ranks(ev0.elapsed_time(ev1) / 1e3, world, dev)

    g_tied = graph_of(B.TQFX4_SRC_F32_TIED)
    with ClockSampler(local) as clk:
        t = timed(g_tied)
    B.tqfx4_check(ws)
    t_rtn = timed(graph_of(B.TQFX4_SRC_F32_RTN))
    B.tqfx4_check(ws)

    # end to end: each matrix from pinned host memory, its blocks back to it
    Wh = [w.cpu().pin_memory() for w in W]
    win = torch.empty((n, k), device=dev)
    outh = torch.empty(out.numel(), dtype=torch.uint8, pin_memory=True)
    for i in range(3):
        win.copy_(Wh[i % PACK_MATS], non_blocking=True)
        B.tqfx4_pack(B.TQFX4_SRC_F32_TIED, win, None, None, n, k, out, ws, stream)
        outh.copy_(out, non_blocking=True)
    torch.cuda.synchronize()
    ev0.record(stream)
    for i in range(args.steps):
        win.copy_(Wh[i % PACK_MATS], non_blocking=True)
        B.tqfx4_pack(B.TQFX4_SRC_F32_TIED, win, None, None, n, k, out, ws, stream)
        outh.copy_(out, non_blocking=True)
    ev1.record(stream)
    torch.cuda.synchronize()
    B.tqfx4_check(ws)
    te = max_over_ranks(ev0.elapsed_time(ev1) / 1e3, world, dev)

    peak, peak_kind = _peaks()
    moved = n * k * 4 + out.numel()  # fp32 in, blocks out
    achieved = moved * args.steps / t / 1e9
    line = {
        "metric": "expert matrices packed per second (tied solver, 2048 x 4096)",
        "value": job_rate(args.steps, world, t), "unit": "matrices/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": t / args.steps * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": "pack_tied", "n": n, "k": k, "matrices_cycled": PACK_MATS,
                   "l2": "inputs larger than L2 (%d MB of fp32 matrices cycled)" % (PACK_MATS * n * k * 4 >> 20)},
        "rtn_same_shape": {"ms_per_step": t_rtn / args.steps * 1e3, "matrices_per_s": args.steps / t_rtn},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                     "traffic": None, "kernel": "pack_kernel (tied source)", "peak_source": peak_kind,
                     "note": "fp32 in + blocks out per launch over its time; the solver (an average of 12.8 "
                             "scale updates a block) is arithmetic-bound, so HBM stays mostly idle"},
        "e2e": {"value": job_rate(args.steps, world, te), "unit": "matrices/s", "h2d_bytes_per_step": n * k * 4,
                "d2h_bytes_per_step": out.numel()},
        "gpu_launches": args.steps,
        "clocks": clk.summary(),
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        rows = 32
        sub = W[0][:rows].cpu().numpy()
        done, el = 0, 0.0
        while el < 10.0:
            t0 = time.perf_counter()
            oracle.pack_tied(sub)
            el += time.perf_counter() - t0
            done += 1
        line["cpu_baseline"] = {"value": done * rows / n / el, "unit": "matrices/s", "cores": 1, "kind": "oracle",
                                "sample": "%d tied packs of the first %d rows, scaled to whole matrices"
                                          % (done, rows)}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()



def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--experts", type=int, default=E,
                    help="routed experts in the layer (default 256; smaller only for profiling captures)")
    ap.add_argument("--tokens", type=int, default=0,
                    help="tokens per step of the grouped workloads (default: 64 or 2048; profiling only)")
    ap.add_argument("--workload", default="moe_decode",
                    choices=["moe_decode", "gemv_1024", "expert_ffn", "grouped_decode_64", "prefill_2048",
                             "tiered_decode", "mxfp4_gemv", "moe_decode_mxfp4", "free_gemv", "pack_tied"],
                    help="moe_decode (default): 1 token; gemv_1024: one 1024 x 1024 GEMV; expert_ffn: one "
                         "SwiGLU expert FFN; grouped_decode_64: 64 tokens with Zipf(1.1) "
                         "routing; prefill_2048: 2048 tokens; tiered_decode: 1 token with the experts in "
                         "host memory; mxfp4_gemv / free_gemv: one GEMV over MXFP4 / free-scale two-plane blocks; "
                         "moe_decode_mxfp4: moe_decode with MXFP4 experts; pack_tied: the tied solver packing expert "
                         "matrices")
    ap.add_argument("--slots", type=int, default=TOPK, help="device expert slots of tiered_decode")
    args = ap.parse_args()
    globals()["E"] = args.experts

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    if args.workload == "tiered_decode":
        run_tiered(args, rank, world, local)
        return
    if args.workload in ("mxfp4_gemv", "free_gemv"):
        run_gemv(args, rank, world, local)
        return
    if args.workload == "pack_tied":
        run_pack(args, rank, world, local)
        return
    if args.workload in ("gemv_1024", "expert_ffn"):
        run_small(args, rank, world, local)
        return
    if args.workload not in ("moe_decode", "moe_decode_mxfp4"):
        run_grouped(args, rank, world, local)
        return
    mx = args.workload == "moe_decode_mxfp4"

    import torch
    import torch.distributed as dist

    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    from paper_2608_08910_gb300 import binding as B
    from paper_2608_08910_gb300 import inputs
    from paper_2608_08910_gb300.moe import MoeLayer

    assert args.warmup >= 3, "at least 3 warm-up steps"
    dev = torch.device("cuda", local)
    layer = (MoeLayer.synthetic_mxfp4 if mx else MoeLayer.synthetic)(SEED, E, H, I, TOPK, 0.0, dev)
    ws = layer.workspace(1)
    X = inputs.hidden_states(SEED + rank, POOL, H, dev)
    out = torch.empty(H, device=dev)
    sel = torch.empty(TOPK, dtype=torch.int32, device=dev)
    selw = torch.empty(TOPK, device=dev)
    stream = torch.cuda.current_stream(dev)
    per_token, gu_bytes, dn_bytes = bytes_per_token(layer)

    def step(i, events=None, st=stream):
        layer.ffn(X[i % POOL], ws, out, sel, selw, stream=st, events=events)

    for i in range(args.warmup):
        step(i)
    B.tqfx4_check(ws)

    # The K steps are captured once into a CUDA graph (the launches keep their
    # programmatic-dependency edges) so that host launch cost stays out of the
    # device timing; each step routes a different hidden state.
    cap_stream = torch.cuda.Stream(dev)
    cap_stream.wait_stream(stream)
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(cap_stream):
        with torch.cuda.graph(graph, stream=cap_stream):
            for i in range(args.steps):
                step(args.warmup + i, st=cap_stream)
    stream.wait_stream(cap_stream)
    graph.replay()  # untimed
    torch.cuda.synchronize()
    B.tqfx4_check(ws)

    # ---- timed region: K steps, device time, max over ranks ----
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clk:
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        ev0.record(stream)
        graph.replay()
        ev1.record(stream)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
    B.tqfx4_check(ws)
    t = ev0.elapsed_time(ev1) / 1e3
    t = max_over_ranks(t, world, dev)
    tokens = args.steps * world  # tokens of the whole job
    value = job_rate(per_token * args.steps, world, t) / 1e9
    # band: five more replays of the same K steps (outside the reported timing)
    reps_ms = []
    for _ in range(5):
        torch.cuda.synchronize()
        ev0.record(stream)
        graph.replay()
        ev1.record(stream)
        torch.cuda.synchronize()
        reps_ms.append(ev0.elapsed_time(ev1) / args.steps)

    # ---- dominant kernel: CUDA events around every stage of every step, on
    # the launching stream (a second graph of the same K steps; the stage
    # launches are plain stream-ordered here) ----
    kind = 2 if mx else 0
    n_st = B.tqfx4_moe_stage_count(kind, 0)
    names = [B.tqfx4_moe_stage_name(kind, 0, s) for s in range(n_st)]
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(n_st + 1)] for _ in range(args.steps)]
    for row in evs:
        for e_ in row:
            e_.record(stream)
    torch.cuda.synchronize()
    graph2 = torch.cuda.CUDAGraph()
    cap_stream.wait_stream(stream)
    with torch.cuda.stream(cap_stream):
        with torch.cuda.graph(graph2, stream=cap_stream):
            for i in range(args.steps):
                step(args.warmup + i, events=evs[i], st=cap_stream)
    stream.wait_stream(cap_stream)
    graph2.replay()
    torch.cuda.synchronize()
    acc = [0.0] * n_st
    for row in evs:
        for s in range(n_st):
            acc[s] += row[s].elapsed_time(row[s + 1]) / 1e3
    stage_s = {names[s]: acc[s] / args.steps for s in range(n_st)}
    dom = "gate_up"
    peak, peak_kind = _peaks()
    achieved = gu_bytes / stage_s[dom] / 1e9

    # ---- end to end through the public API with host buffers ----
    # (fx4: tqfx4_moe_ffn_host, one call a token that copies x in and the
    # output and selection out on the stream; MXFP4: torch copies around the
    # device call)
    Xh = X.cpu().pin_memory()
    outh = torch.empty(H, pin_memory=True)
    selh = torch.empty(TOPK, dtype=torch.int32, pin_memory=True)
    if mx:
        xin = torch.empty(H, device=dev)

        def e2e_step(i):
            xin.copy_(Xh[i], non_blocking=True)
            layer.ffn(xin, ws, out, sel, selw, stream=stream)
            outh.copy_(out, non_blocking=True)
            selh.copy_(sel, non_blocking=True)
        ws_e = ws
    else:
        ws_e = layer.host_workspace()

        def e2e_step(i):
            layer.ffn_host(Xh[i], ws_e, outh, selh, None, stream=stream)
    for i in range(3):
        e2e_step(i)
    torch.cuda.synchronize()
    ev0.record(stream)
    for i in range(args.steps):
        e2e_step(i % POOL)
    ev1.record(stream)
    torch.cuda.synchronize()
    B.tqfx4_check(ws_e)
    te = ev0.elapsed_time(ev1) / 1e3
    te = max_over_ranks(te, world, dev)
    e2e = per_token * tokens / te / 1e9

    line = {
        "metric": METRIC_MX if mx else METRIC, "value": value, "unit": "GB/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": t / args.steps * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "i8xe2m1-i32,f32" if mx else "i8xi4-i32,f32",
        "data": "synthetic",
        "config": {"workload": WORKLOAD_MX if mx else WORKLOAD, "experts": E, "hidden": H, "inter": I,
                   "top_k": TOPK, "tokens_per_step": 1, "bytes_per_token": per_token,
                   "l2": "inputs larger than L2: %.2f GB expert pool, a different hidden state per step"
                         % ((2 * layer.mb_gu + layer.mb_d) * E / 1e9),
                   "parallelism": "replicas" if world > 1 else "single"},
        "tokens_per_s": tokens / t,
        "pct_of_hbm_peak": 100.0 * value / peak,
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": None if mx else GATE_UP_TRAFFIC,
                     "kernel": "mxfp4_gemv_kernel (gate_up)" if mx else dom,
                     "algorithmic_bytes": gu_bytes,
                     "traffic_source": "ncu capture (dram__bytes_read + write) of one gate_up_kernel launch",
                     "peak_source": peak_kind + " (MEASURED_PEAKS.json hbm_gbs)" if peak_kind == "measured"
                     else "fallback 6.8 TB/s",
                     "stage_us": {k: v * 1e6 for k, v in stage_s.items()}},
        "e2e": {"value": e2e, "unit": "GB/s", "h2d_bytes_per_step": H * 4,
                "d2h_bytes_per_step": H * 4 + TOPK * 4},
        # router, gate_up, down (tq2_0_fx4); router, gate_up, down, combine (MXFP4)
        "gpu_launches": (4 if mx else 3) * args.steps,
        "clocks": clk.summary(),
        "repeats_ms_per_step": {"min": min(reps_ms), "median": statistics.median(reps_ms), "max": max(reps_ms),
                                "spread": (max(reps_ms) - min(reps_ms)) / statistics.median(reps_ms),
                                "n": len(reps_ms), "note": "5 more replays of the timed graph"},
    }
    if rank == 0 and not args.no_cpu_baseline:
        v, n, secs = cpu_baseline(layer=layer if mx else None)
        line["cpu_baseline"] = {"value": v, "unit": "GB/s", "cores": 1, "kind": "oracle",
                                "sample": "%d tokens through the layer (%.1f s), expert packing excluded" % (n, secs)}
        if world == 1 and not mx:
            va, na, sa, ca = cpu_baseline_all_cores()
            line["cpu_baseline_all_cores"] = {
                "value": va, "unit": "GB/s", "cores": ca, "kind": "oracle",
                "sample": "%d tokens on %d threads (%.1f s wall), expert packing excluded" % (na, ca, sa)}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
