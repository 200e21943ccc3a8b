"""Benchmark of the per-head-window KV decode path on GB300.

One step = one decode step of every layer of the workload: for each layer,
hwkv_decode_step appends the new token's K/V into every KV head's ring and runs
the split-KV decode attention of all query heads over the resident rings with
the log-sum-exp combine (two launches), plus the residency query
(hwkv_residency_bytes). Inputs are seeded synthetic bf16 tensors from
hwkv_gen with the workload's shapes; the prompt is filled (untimed) before.

Prints one JSON line. `value` is decode tokens/s of the whole job (batch rows
x steps / max-over-ranks time), inputs resident in HBM; `e2e` is the same
metric with each step's q/k/v copied from pinned host memory and the outputs
read back inside the timed region. `roofline` rates the decode kernel against
the measured HBM copy bandwidth; `prefill` reports the window-limited prefill
in TFLOP/s (64K prompt in 8K chunks at head_dim 128, over bf16 and 8-bit caches,
and a 32K prompt at head_dim 256); `append` rates hwkv_append of 8K-token chunks
against the copy bandwidth; `cpu_baseline` is the fp64 oracle on a bounded sample,
on the host cores.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
    python bench.py --impl reference ...   # the oracle arm, on host cores
"""
import argparse
import json
import os
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from hwkv_gen import workloads  # noqa: E402

NOMINAL_HBM_GBS = 8000.0
L2_BYTES = 129 * 1024 * 1024
# DRAM bytes (read + write) per algorithmic byte of the decode split kernel, from an ncu
# capture (--set full) of the 1-layer, batch-2 case of layers16_112k
# (profiles/decode_split_small_full.md); traffic is reads of every resident K/V row plus
# segment partials, so it scales with the algorithmic bytes of a launch. Set to None
# whenever that kernel changes.
DECODE_TRAFFIC_PER_BYTE = (244.291584e6 + 4.332032e6) / 244064256.0
# tensor-pipe activity of the prefill kernel (ncu sm__pipe_tensor_cycles_active, pct of peak
# sustained active) from the one-launch --set full capture summarised in the named profile;
# set to None whenever that kernel changes.
PREFILL_TENSOR_PIPE = {"prefill64k": (0.512, "profiles/prefill_tc_prefill64k_full.md")}


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        d = json.load(open(p))
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), float(
            d.get("bf16_tflops_sustained", d["bf16_tflops"])), "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


# ------------------------------------------------------------------ ranks
def dist_setup(n_gpus):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = os.environ.get("HWKV_BENCH_BACKEND", "nccl")
        if backend == "nccl":
            import torch
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x, world):
    """Max of a float over all ranks (the job's time is its slowest rank)."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(x, world):
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


# ----------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            import tempfile
            fd, self.path = tempfile.mkstemp(prefix="hwkv_clocks_", suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if not self.path or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        rows = []
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) >= 9:
                try:
                    rows.append((float(f[1]), float(f[2]), f[5:9]))
                except ValueError:
                    pass
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, r in rows for i, v in enumerate(r)
                          if v.lower().startswith("active")})
        sm = sorted(r[0] for r in rows)
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


# ------------------------------------------------------------ GPU decode
def token_bytes(wl, fp8=False):
    """Bytes one resident token of one KV head occupies: K and V rows in bf16, or
    E4M3 codes plus a 4-byte scale per row."""
    return 2 * (wl.head_dim + 4) if fp8 else 4 * wl.head_dim


def decode_bytes(wl, max_ctx, t, fp8=False):
    """Algorithmic bytes of one decode launch per layer at length t: every
    resident K/V row read once, batch x sum_h min(t, cap_h) x token_bytes (q and
    out are under 0.1 % and excluded)."""
    per_layer = []
    for layer in range(wl.n_layers):
        s = 0
        for h in range(wl.n_kv_heads):
            W = wl.windows[layer * wl.n_kv_heads + h]
            cap = max_ctx if (W == 0 or W >= max_ctx) else W
            s += wl.batch * min(t, cap) * token_bytes(wl, fp8)
        per_layer.append(s)
    return per_layer


def run_gpu(args, wl, world, rank, local, fp8=False):
    import torch

    import hwkv_gen
    import paper_2609_02029_gb300 as hwkv

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    hwkv.lib()
    stream = torch.cuda.current_stream(dev)  # every allocation and launch on one stream
    s = stream.cuda_stream
    g = hwkv_gen.desc(wl.seed + 1000003 * rank, wl.per_head_scale)  # each rank its own batch
    L, B, Hq, Hkv, d = wl.n_layers, wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim
    e2e_steps = min(args.steps, args.e2e_steps)
    graph_steps = min(args.steps, 32)
    total_steps = args.warmup + args.steps + 2 + e2e_steps + 3 + graph_steps
    prompt = wl.prompt
    max_ctx = prompt + max(wl.decode_steps, total_steps)
    scale = 1.0 / np.sqrt(d)

    pol = hwkv.make_policy(L, Hkv, Hq, d, B, max_ctx, wl.windows,
                           kv_format=hwkv.HWKV_KV_FP8_E4M3 if fp8 else hwkv.HWKV_KV_BF16)
    nbytes = hwkv.hwkv_required_bytes(pol)
    arena = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    cache = hwkv.hwkv_alloc(pol, arena, nbytes, s)

    # prompt fill (untimed): generated chunks appended through the C ABI
    chunk = 4096
    kbuf = torch.empty((B, chunk, Hkv, d), dtype=torch.bfloat16, device=dev)
    vbuf = torch.empty_like(kbuf)
    for layer in range(L):
        done = 0
        while done < prompt:
            n = min(chunk, prompt - done)
            hwkv_gen.fill_device(g, hwkv_gen.K, layer, B, done, n, Hkv, d, kbuf.data_ptr(), s)
            hwkv_gen.fill_device(g, hwkv_gen.V, layer, B, done, n, Hkv, d, vbuf.data_ptr(), s)
            hwkv.hwkv_append(cache, layer, kbuf, vbuf, n, s)
            done += n
    del kbuf, vbuf

    # per-step inputs (q of the new token, its K/V), pre-generated on the device
    def gen_step(pos):
        q = torch.empty((L, B, Hq, d), dtype=torch.bfloat16, device=dev)
        k = torch.empty((L, B, 1, Hkv, d), dtype=torch.bfloat16, device=dev)
        v = torch.empty_like(k)
        for layer in range(L):
            hwkv_gen.fill_device(g, hwkv_gen.Q, layer, B, pos, 1, Hq, d, q[layer].data_ptr(), s)
            hwkv_gen.fill_device(g, hwkv_gen.K, layer, B, pos, 1, Hkv, d, k[layer].data_ptr(), s)
            hwkv_gen.fill_device(g, hwkv_gen.V, layer, B, pos, 1, Hkv, d, v[layer].data_ptr(), s)
        return q, k, v

    n_dev = args.warmup + args.steps
    inputs = [gen_step(prompt + i) for i in range(n_dev)]
    out = torch.empty((L, B, Hq, d), dtype=torch.float32, device=dev)
    stream.synchronize()

    # per-launch events on layer 0 of every step only: events between launches would
    # also stop the next launch from overlapping its predecessor's tail
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True),
           torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    resid = []
    # a layer-step that reads less than twice the L2 would run from L2 on repeats:
    # then every timed step is preceded by a read of a 2 x L2 buffer, outside its
    # events (a read leaves clean lines, so no write-back competes with the step)
    flush = max(decode_bytes(wl, max_ctx, prompt + 1, fp8)) < 2 * L2_BYTES
    scrub = torch.ones(2 * L2_BYTES // 4, dtype=torch.float32, device=dev) if flush else None
    scrub_out = torch.empty((), dtype=torch.float32, device=dev) if flush else None
    step_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(args.steps)]

    def step(i, timed_idx=None):
        q, k, v = inputs[i]
        for layer in range(L):
            mark = timed_idx is not None and layer == 0
            if mark:
                ev[timed_idx][0].record(stream)
                ev[timed_idx][1].record(stream)
            hwkv.hwkv_decode_step(cache, layer, q[layer], k[layer], v[layer], scale, out[layer], s)
            if mark:
                ev[timed_idx][2].record(stream)
        resid.append(hwkv.hwkv_residency_bytes(cache, -1))

    for i in range(args.warmup):
        step(i)
    t_first = hwkv.hwkv_seq_len(cache, 0)
    stream.synchronize()
    barrier(world)
    torch.cuda.synchronize()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clk:
        start.record(stream)
        for j in range(args.steps):
            if flush:
                torch.sum(scrub, dim=0, out=scrub_out)
            step_ev[j][0].record(stream)
            step(args.warmup + j, j)
            step_ev[j][1].record(stream)
        end.record(stream)
        end.synchronize()
    torch.cuda.synchronize()
    barrier(world)
    ms_local = (sum(a.elapsed_time(b) for a, b in step_ev) if flush
                else start.elapsed_time(end))
    clocks = clk.summary()
    hwkv.hwkv_sync_check(cache)

    # decode launch durations (layer 0 of every timed step) and their algorithmic bytes
    dec_ms, app_ms, dec_bytes, step_bytes = [], [], [], []
    for j in range(args.steps):
        t = t_first + j + 1
        per_layer = decode_bytes(wl, max_ctx, t, fp8)
        e0, e1, e2 = ev[j]
        app_ms.append(e0.elapsed_time(e1))
        dec_ms.append(e1.elapsed_time(e2))
        dec_bytes.append(per_layer[0])
        step_bytes.append(sum(per_layer))
    dec_avg_ms = float(np.mean(dec_ms))
    bytes_avg = float(np.mean(dec_bytes))
    achieved_gbs = bytes_avg / (dec_avg_ms * 1e-3) / 1e9
    step_bytes = float(np.mean(step_bytes))

    ms = max_over_ranks(ms_local, world)
    tokens = sum_over_ranks(float(B * args.steps), world)
    value = tokens / (ms * 1e-3)

    # ---- end to end: host inputs in, host outputs out, every step
    o_h = torch.empty((L, B, Hq, d), dtype=torch.float32, pin_memory=True)
    q_d = torch.empty((L, B, Hq, d), dtype=torch.bfloat16, device=dev)
    k_d = torch.empty((L, B, 1, Hkv, d), dtype=torch.bfloat16, device=dev)
    v_d = torch.empty_like(k_d)
    pos0 = hwkv.hwkv_seq_len(cache, 0)
    host_inputs = []
    for i in range(e2e_steps + 2):
        q, k, v = gen_step(pos0 + i)
        host_inputs.append((q.cpu().pin_memory(), k.cpu().pin_memory(), v.cpu().pin_memory()))
    stream.synchronize()

    # Copies overlap the decode: a copy stream brings layer l's q/k/v in while
    # earlier layers decode, another takes layer l's output out while later ones
    # run; the step ends when the last output has reached the host. The next
    # step's copies start only after this step's end (they reuse the buffers).
    copy_in, copy_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    ev_in = [torch.cuda.Event() for _ in range(L)]
    ev_out = [torch.cuda.Event() for _ in range(L)]
    ev_start, ev_done = torch.cuda.Event(), torch.cuda.Event()

    def e2e_step(i):
        qh, kh, vh = host_inputs[i]
        ev_start.record(stream)
        copy_in.wait_event(ev_start)
        with torch.cuda.stream(copy_in):
            for layer in range(L):
                q_d[layer].copy_(qh[layer], non_blocking=True)
                k_d[layer].copy_(kh[layer], non_blocking=True)
                v_d[layer].copy_(vh[layer], non_blocking=True)
                ev_in[layer].record(copy_in)
        for layer in range(L):
            stream.wait_event(ev_in[layer])
            hwkv.hwkv_decode_step(cache, layer, q_d[layer], k_d[layer], v_d[layer], scale,
                                  out[layer], s)
            ev_out[layer].record(stream)
            copy_out.wait_event(ev_out[layer])
            with torch.cuda.stream(copy_out):
                o_h[layer].copy_(out[layer], non_blocking=True)
        ev_done.record(copy_out)
        stream.wait_event(ev_done)

    for i in range(2):
        e2e_step(i)
    stream.synchronize()
    barrier(world)
    e2e_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(e2e_steps)]
    for i in range(e2e_steps):
        if flush:
            torch.sum(scrub, dim=0, out=scrub_out)
        e2e_ev[i][0].record(stream)
        e2e_step(2 + i)
        e2e_ev[i][1].record(stream)
    e2e_ev[-1][1].synchronize()
    barrier(world)
    e2e_ms = max_over_ranks(sum(a.elapsed_time(b) for a, b in e2e_ev), world)
    e2e_value = sum_over_ranks(float(B * e2e_steps), world) / (e2e_ms * 1e-3)
    h2d = int(sum(x.numel() * x.element_size() for x in host_inputs[0]))
    d2h = int(o_h.numel() * 4)

    # ---- the same step as one captured CUDA graph of hwkv_decode_step_graph calls
    # (device-side lengths and tile plan), replayed; inputs refilled between replays
    pos = hwkv.hwkv_seq_len(cache, 0)
    stream.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        cs = torch.cuda.current_stream().cuda_stream
        for layer in range(L):
            hwkv.hwkv_decode_step_graph(cache, layer, q_d[layer], k_d[layer], v_d[layer], scale,
                                        out[layer], cs)

    def graph_inputs(p):
        for layer in range(L):
            hwkv_gen.fill_device(g, hwkv_gen.Q, layer, B, p, 1, Hq, d, q_d[layer].data_ptr(), s)
            hwkv_gen.fill_device(g, hwkv_gen.K, layer, B, p, 1, Hkv, d, k_d[layer].data_ptr(), s)
            hwkv_gen.fill_device(g, hwkv_gen.V, layer, B, p, 1, Hkv, d, v_d[layer].data_ptr(), s)

    for i in range(3):
        graph_inputs(pos)
        graph.replay()
        pos += 1
    g_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
            for _ in range(graph_steps)]
    for i in range(graph_steps):
        graph_inputs(pos)
        if flush:
            torch.sum(scrub, dim=0, out=scrub_out)
        g_ev[i][0].record(stream)
        graph.replay()
        g_ev[i][1].record(stream)
        pos += 1
    g_ev[-1][1].synchronize()
    graph_ms = max_over_ranks(sum(a.elapsed_time(b) for a, b in g_ev), world)
    graph_value = sum_over_ranks(float(B * graph_steps), world) / (graph_ms * 1e-3)
    del graph
    t_end = hwkv.hwkv_seq_len(cache, 0)  # re-read from the device (graph-owned layers)
    assert t_end == pos, (t_end, pos)
    resid_bytes = hwkv.hwkv_residency_bytes(cache, -1)
    hwkv.hwkv_sync_check(cache)
    hwkv.hwkv_free(cache)
    del arena, inputs
    torch.cuda.empty_cache()

    return dict(value=value, ms=ms, e2e_value=e2e_value, e2e_ms=e2e_ms, h2d=h2d, d2h=d2h,
                dec_avg_ms=dec_avg_ms, app_avg_ms=float(np.mean(app_ms)), bytes_avg=bytes_avg,
                achieved_gbs=achieved_gbs, step_bytes=step_bytes, clocks=clocks,
                t_first=t_first, t_end=t_end, resid_bytes=resid_bytes,
                launches=args.steps * L * 2, e2e_steps=e2e_steps, max_ctx=max_ctx, flush=flush,
                steps=args.steps,
                graph_value=graph_value, graph_ms=graph_ms, graph_steps=graph_steps)


SECONDARY_WORKLOADS = ["tiny", "single32k", "budget161k_r25", "budget161k_r50",
                       "budget161k_r75", "budget161k_r100"]


def workload_by_name(name):
    if name.startswith("budget161k_r"):
        return workloads.make("budget161k", int(name.split("_r")[1]) / 100.0)
    return workloads.make(name)


def run_secondary(args, name, world, rank, local, hbm):
    """The same decode step on another workload (fewer timed steps): device-timed
    tokens/s, the replayed-graph form, end to end, and the decode call's rate
    against the copy bandwidth."""
    wl = workload_by_name(name)
    a = argparse.Namespace(**vars(args))
    a.steps, a.e2e_steps = min(args.steps, 32), min(args.e2e_steps, 8)
    r = run_gpu(a, wl, world, rank, local)
    graph_gbs = r["step_bytes"] / (r["graph_ms"] / r["graph_steps"] * 1e-3) / 1e9
    return {"workload": wl.name, "layers": wl.n_layers, "batch_per_gpu": wl.batch,
            "head_dim": wl.head_dim, "context": wl.max_ctx, "windows": wl.note,
            "value": r["value"], "unit": "tokens/s", "steps": a.steps,
            "ms_per_step": r["ms"] / a.steps,
            "graph_value": r["graph_value"], "graph_ms_per_step": r["graph_ms"] / r["graph_steps"],
            "e2e_value": r["e2e_value"],
            "decode_gbs": r["achieved_gbs"], "frac": r["achieved_gbs"] / hbm,
            "bytes_per_launch": r["bytes_avg"], "launch_ms": r["dec_avg_ms"],
            "step_bytes": r["step_bytes"],
            "graph_step_gbs": graph_gbs,
            # the whole replayed step (every layer's split and combine launches) against
            # the copy bandwidth; frac above is one eager layer launch
            "graph_frac": graph_gbs / hbm,
            "l2": ("each timed step preceded by a 2 x L2 read outside its events"
                   if r["flush"] else "inputs larger than L2"),
            "residency_bytes": r["resid_bytes"]}


# ------------------------------------------------------------- GPU prefill
def prefill_flops(wl, t0, n):
    """Algorithmic flops of one prefill chunk: 4 d G per visible (query, key) pair."""
    total = 0
    for h in range(wl.n_kv_heads):
        W = wl.windows[h]
        # visible keys of query p: min(p + 1, W) (full: p + 1); sum over p in the chunk
        if W == 0 or W >= wl.max_ctx:
            pairs = sum_range(t0 + 1, t0 + n)
        else:
            lo, hi = t0 + 1, t0 + n  # p + 1 ranges over [lo, hi]
            cut = min(max(W, lo - 1), hi)  # p + 1 <= W counts p + 1, above counts W
            pairs = sum_range(lo, cut) + W * (hi - cut)
        total += pairs * wl.group * 4 * wl.head_dim * wl.batch
    return total


def sum_range(a, b):
    """a + (a+1) + ... + b (0 if b < a)."""
    return 0 if b < a else (a + b) * (b - a + 1) // 2


def run_prefill(args, local, fp8=False, workload="prefill64k"):
    """A whole prompt in 8,192-token chunks through hwkv_prefill: prefill64k (64K
    tokens, head_dim 128) or single32k (32K tokens, head_dim 256). With fp8 the cache
    holds E4M3 codes + row scales; the timed region then also covers the per-call
    staging of the visible rows and the 8-bit append."""
    import torch

    import hwkv_gen
    import paper_2609_02029_gb300 as hwkv

    wl = workloads.make(workload)
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream(dev)
    s = stream.cuda_stream
    g = hwkv_gen.desc(wl.seed, wl.per_head_scale)
    B, Hq, Hkv, d, n = wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.chunk
    chunks = wl.prompt // n
    scale = 1.0 / np.sqrt(d)
    q = torch.empty((chunks, B, n, Hq, d), dtype=torch.bfloat16, device=dev)
    k = torch.empty((chunks, B, n, Hkv, d), dtype=torch.bfloat16, device=dev)
    v = torch.empty_like(k)
    for c in range(chunks):
        hwkv_gen.fill_device(g, hwkv_gen.Q, 0, B, c * n, n, Hq, d, q[c].data_ptr(), s)
        hwkv_gen.fill_device(g, hwkv_gen.K, 0, B, c * n, n, Hkv, d, k[c].data_ptr(), s)
        hwkv_gen.fill_device(g, hwkv_gen.V, 0, B, c * n, n, Hkv, d, v[c].data_ptr(), s)
    out = torch.empty((B, n, Hq, d), dtype=torch.float32, device=dev)
    pol = hwkv.make_policy(1, Hkv, Hq, d, B, wl.max_ctx, wl.windows,
                           kv_format=hwkv.HWKV_KV_FP8_E4M3 if fp8 else hwkv.HWKV_KV_BF16)
    nbytes = hwkv.hwkv_required_bytes(pol)
    arena = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    reps = []
    flops = sum(prefill_flops(wl, c * n, n) for c in range(chunks))
    warm = 3 if args.prefill_reps > 1 else 1  # a single rep is the profiling case
    for rep in range(warm + args.prefill_reps):
        cache = hwkv.hwkv_alloc(pol, arena, nbytes, s)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for c in range(chunks):
            hwkv.hwkv_prefill(cache, 0, q[c], k[c], v[c], n, scale, out, s)
        e1.record(stream)
        e1.synchronize()
        hwkv.hwkv_sync_check(cache)
        hwkv.hwkv_free(cache)
        if rep >= warm:
            reps.append(e0.elapsed_time(e1))
    ms = float(np.median(reps))
    del q, k, v, out, arena
    torch.cuda.empty_cache()
    return dict(ms=ms, flops=flops, tflops=flops / (ms * 1e-3) / 1e12,
                tokens_per_s=B * wl.prompt / (ms * 1e-3))


# ------------------------------------------------------------ GPU append
def run_append(local, n=8192, reps=8, warm=3, fp8=False, batch=0):
    """hwkv_append of 8,192-token chunks into layer 0 of layers16_112k (batch 16,
    4 KV heads, d 256, rings of {full, 32768, 8192, 2048, 512} drawn per head):
    each call reads the chunk's K and V (537 MB, more than L2) and writes the last
    min(n, cap) tokens of every head into its ring. Algorithmic bytes per call:
    batch x sum_h min(n, cap_h) x 4d written plus the same read from the input
    (only the rows that land are read). Full heads hold max_ctx = 14 chunks, so at
    most 14 calls. With fp8 the cache holds E4M3 codes + one fp32 scale per row: bytes
    per landing row and head are the bf16 K and V read (4d) plus codes and scales
    written (2d + 8)."""
    import torch

    import hwkv_gen
    import paper_2609_02029_gb300 as hwkv

    wl = workloads.make("layers16_112k")
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream(dev)
    s = stream.cuda_stream
    g = hwkv_gen.desc(wl.seed, wl.per_head_scale)
    B, Hkv, d = (batch or wl.batch), wl.n_kv_heads, wl.head_dim
    windows = wl.windows[:Hkv]
    k = torch.empty((B, n, Hkv, d), dtype=torch.bfloat16, device=dev)
    v = torch.empty_like(k)
    hwkv_gen.fill_device(g, hwkv_gen.K, 0, B, 0, n, Hkv, d, k.data_ptr(), s)
    hwkv_gen.fill_device(g, hwkv_gen.V, 0, B, 0, n, Hkv, d, v.data_ptr(), s)
    pol = hwkv.make_policy(1, Hkv, wl.n_q_heads, d, B, wl.max_ctx, windows,
                           kv_format=hwkv.HWKV_KV_FP8_E4M3 if fp8 else hwkv.HWKV_KV_BF16)
    nbytes = hwkv.hwkv_required_bytes(pol)
    arena = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    cache = hwkv.hwkv_alloc(pol, arena, nbytes, s)
    caps = [wl.max_ctx if (W == 0 or W >= wl.max_ctx) else W for W in windows]
    per_row = (4 * d + 2 * d + 8) if fp8 else 2 * 4 * d
    per_call = B * sum(min(n, c) for c in caps) * per_row
    # the full heads hold max_ctx = 14 chunks: warm-up calls, then `reps` calls back to back
    # between one pair of events (the chunks of a prompt arrive that way; the host's launch
    # path overlaps the previous call), then single calls each between its own events
    singles = max(0, min(4, wl.max_ctx // n - warm - reps))
    for _ in range(warm):
        hwkv.hwkv_append(cache, 0, k, v, n, s)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize(dev)
    e0.record(stream)
    for _ in range(reps):
        hwkv.hwkv_append(cache, 0, k, v, n, s)
    e1.record(stream)
    e1.synchronize()
    ms = e0.elapsed_time(e1) / reps
    single = []
    for _ in range(singles):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        hwkv.hwkv_append(cache, 0, k, v, n, s)
        b.record(stream)
        b.synchronize()
        single.append(a.elapsed_time(b))
    hwkv.hwkv_sync_check(cache)
    hwkv.hwkv_free(cache)
    del k, v, arena
    torch.cuda.empty_cache()
    return {"workload": "layers16_112k layer 0, 8192-token chunks" + (", 8-bit cache" if fp8 else "")
                        + (", batch %d" % B if batch else ""),
            "ms": ms, "calls_timed": reps,
            "single_call_ms": float(np.median(single)) if single else None,
            "bytes_per_call": per_call, "gbs": per_call / (ms * 1e-3) / 1e9}


# ------------------------------------------------------------ GPU SeqCalib
def run_calib(local, T=131072, P=256, Hkv=4, Hq=24, d=256, windows=(8192, 16384, 32768), reps=3):
    """Candidate replay of one layer's trace: a T-token trace, P query positions
    drawn from its final quarter, every candidate window scored against full.
    Algorithmic bytes: each (position, KV head) reads its t + 1 keys once (4 d B)."""
    import torch

    import hwkv_gen
    import paper_2609_02029_gb300 as hwkv

    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream(dev)
    s = stream.cuda_stream
    g = hwkv_gen.desc(7)
    rng = np.random.default_rng(3)
    pos = np.sort(rng.choice(np.arange(T - T // 4, T), size=P, replace=False))[None, :]
    K = torch.empty((1, T, Hkv, d), dtype=torch.bfloat16, device=dev)
    V = torch.empty_like(K)
    hwkv_gen.fill_device(g, hwkv_gen.K, 0, 1, 0, T, Hkv, d, K.data_ptr(), s)
    hwkv_gen.fill_device(g, hwkv_gen.V, 0, 1, 0, T, Hkv, d, V.data_ptr(), s)
    Kh = K.permute(0, 2, 1, 3).contiguous()
    Vh = V.permute(0, 2, 1, 3).contiguous()
    del K, V
    q = torch.empty((1, P, Hq, d), dtype=torch.bfloat16, device=dev)
    for i in range(P):
        hwkv_gen.fill_device(g, hwkv_gen.Q, 0, 1, int(pos[0, i]), 1, Hq, d, q[0, i].data_ptr(), s)
    desc = hwkv.make_calib_desc(1, P, Hkv, Hq, d, T, list(windows), pos)
    nbytes = hwkv.hwkv_calib_workspace_bytes(desc)
    ws = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    scale = 1.0 / np.sqrt(d)
    times = []
    for rep in range(reps + 1):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        scores, _ = hwkv.hwkv_calib_scores(desc, q, Kh, Vh, scale, ws, nbytes, stream)
        t1 = time.perf_counter()  # the call synchronizes its stream
        if rep:
            times.append(t1 - t0)
    sec = float(np.median(times))
    keys = int((pos + 1).sum()) * Hkv
    del Kh, Vh, q, ws
    torch.cuda.empty_cache()
    return {"trace_tokens": T, "positions": P, "kv_heads": Hkv, "q_heads": Hq, "head_dim": d,
            "windows": list(windows), "ms": sec * 1e3, "keys_replayed": keys,
            "gbs": keys * 4 * d / sec / 1e9, "positions_per_s": P / sec,
            "mean_scores": [float(x) for x in scores.mean(axis=0)],
            "note": "wall time of hwkv_calib_scores (plan, upload, both kernels, readback)"}


# ------------------------------------------------------------ CPU oracle
def step_keys(wl, max_ctx, t):
    """(layer, batch row, KV head) units of one decode step at length t and the
    keys each attends to."""
    out = []
    for l in range(wl.n_layers):
        for h in range(wl.n_kv_heads):
            W = wl.windows[l * wl.n_kv_heads + h]
            cap = max_ctx if (W == 0 or W >= max_ctx) else W
            for b in range(wl.batch):
                out.append((l, b, h, W if cap == W else 0, min(t, cap)))
    return out


class OracleLayerSteps:
    """The fp64 oracle (array form) over whole layer-steps of the decode: for one
    layer at position p, every (batch row, KV head) unit's G queries over all of
    its retained keys. A layer's inputs are generated on the host before its clock
    starts (one unit per thread); then the oracle runs over every unit of the layer
    with all host cores busy (one unit per thread, one OpenMP thread each), largest
    units first, and only that is timed."""

    def __init__(self, wl, max_ctx):
        self.wl, self.max_ctx = wl, max_ctx
        self.cores = os.cpu_count() or 1
        self.units_per_layer = wl.batch * wl.n_kv_heads

    def _inputs(self, layer, p):
        from concurrent.futures import ThreadPoolExecutor

        import hwkv_gen
        import oracle

        wl = self.wl
        g = hwkv_gen.desc(wl.seed, wl.per_head_scale)
        d, G = wl.head_dim, wl.group
        units = []
        for h in range(wl.n_kv_heads):
            W = wl.windows[layer * wl.n_kv_heads + h]
            Weff = 0 if (W == 0 or W >= self.max_ctx) else W
            for b in range(wl.batch):
                units.append((b, h, Weff))

        def make(u):
            b, h, W = u
            lo = oracle.window_lo(p, W)
            K = hwkv_gen.fill_host_sub(g, hwkv_gen.K, layer, b, lo, p - lo + 1, h, 1, d)[:, 0]
            V = hwkv_gen.fill_host_sub(g, hwkv_gen.V, layer, b, lo, p - lo + 1, h, 1, d)[:, 0]
            Q = hwkv_gen.fill_host_sub(g, hwkv_gen.Q, layer, b, p, 1, h * G, G, d)[0]
            return (Q, K, V, p - lo)

        with ThreadPoolExecutor(max_workers=self.cores) as ex:
            inputs = list(ex.map(make, units))
        inputs.sort(key=lambda x: -x[1].shape[0])
        return inputs

    def run_layer(self, layer, p):
        """(seconds, units, keys) of the oracle over every unit of `layer` at position p."""
        import threading
        from concurrent.futures import ThreadPoolExecutor

        import oracle

        inputs = self._inputs(layer, p)
        local = threading.local()
        gamma = 1.0 / np.sqrt(self.wl.head_dim)

        def work(u):
            if not getattr(local, "set", False):
                oracle.set_threads(1)
                local.set = True
            Q, K, V, p_rel = u
            oracle.window_attention_bf16(Q, [p_rel] * len(Q), K, V, 0, gamma)

        with ThreadPoolExecutor(max_workers=self.cores) as ex:
            t0 = time.perf_counter()
            list(ex.map(work, inputs))
            sec = time.perf_counter() - t0
        return sec, len(inputs), sum(x[1].shape[0] for x in inputs)


def cpu_baseline(wl, max_ctx, t, steps=2):
    """Oracle tokens/s on this host's cores over `steps` whole decode steps (every
    layer, batch row and KV head) at positions t - 1, t, ...; input generation is
    outside the timed part."""
    orc = OracleLayerSteps(wl, max_ctx)
    sec, units, keys = 0.0, 0, 0
    for st in range(steps):
        for layer in range(wl.n_layers):
            s_, u_, k_ = orc.run_layer(layer, t - 1 + st)
            sec += s_
            units += u_
            keys += k_
    return {"value": wl.batch * steps / sec, "unit": "tokens/s", "cores": orc.cores,
            "kind": "oracle", "seconds": sec,
            "sample": "%d whole decode steps at t=%d..%d: all %d (layer, batch row, KV head) "
                      "units each, %d keys in all; fp64 oracle %.1f s on %d threads (input "
                      "generation before each layer's clock, not timed)"
                      % (steps, t, t + steps - 1, units // steps, keys, sec, orc.cores)}


# ------------------------------------------------------------------ main
def emit(obj):
    print(json.dumps(obj), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=96)
    ap.add_argument("--warmup", type=int, default=4)
    ap.add_argument("--workload", default="layers16_112k",
                    choices=["layers16_112k", "single32k", "budget161k_r25", "budget161k_r50",
                             "budget161k_r75", "budget161k_r100"])
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--e2e-steps", type=int, default=32)
    ap.add_argument("--kv", choices=["bf16", "fp8"], default="bf16",
                    help="cache format of the timed decode (fp8: E4M3 codes + row scales)")
    ap.add_argument("--no-fp8", action="store_true",
                    help="skip the secondary 8-bit-cache decode measurement")
    ap.add_argument("--prefill-reps", type=int, default=5)
    ap.add_argument("--no-prefill", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-calib", action="store_true")
    ap.add_argument("--no-secondary", action="store_true",
                    help="skip the decode lines of the other workloads (tiny, single32k, the "
                         "161K budget sweep)")
    ap.add_argument("--prefill-only", action="store_true",
                    help="run only a prefill measurement (profiling)")
    ap.add_argument("--append-only", action="store_true",
                    help="run only the chunk append measurement (profiling)")
    ap.add_argument("--prefill-workload", default="prefill64k", choices=["prefill64k", "single32k"],
                    help="prompt of --prefill-only")
    ap.add_argument("--layers", type=int, default=0,
                    help="profiling only: keep the first N layers (the reported workload is "
                         "the full one)")
    ap.add_argument("--batch", type=int, default=0, help="profiling only: batch rows")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")

    if args.workload.startswith("budget161k_r"):
        wl = workloads.make("budget161k", int(args.workload.split("_r")[1]) / 100.0)
    else:
        wl = workloads.make(args.workload)
    if args.layers:
        wl.n_layers = args.layers
        wl.windows = wl.windows[:args.layers * wl.n_kv_heads]
        wl.name += "_L%d" % args.layers
    if args.batch:
        wl.batch = args.batch
        wl.name += "_B%d" % args.batch
    hbm, tf_burst, tf_sust, peak_src = peaks()
    world, rank, local = dist_setup(args.gpus)
    metric = "decode attn tokens/s on per-head-window KV"
    config = {"workload": wl.name, "layers": wl.n_layers, "batch_per_gpu": wl.batch,
              "q_heads": wl.n_q_heads, "kv_heads": wl.n_kv_heads, "head_dim": wl.head_dim,
              "context": wl.max_ctx, "window_levels": wl.levels, "note": wl.note,
              "parallelism": "replicas" if args.gpus > 1 else "single",
              "l2": "inputs larger than L2", "kv_format": args.kv}

    if args.impl == "reference":
        if rank != 0:
            return
        # each step = the decode of `lps` layers (all batch rows and KV heads) by the fp64
        # oracle on the host cores: lps / L of a whole decode step, so the steps cover
        # whole decode steps (L / lps steps each) at advancing positions
        lps = max(1, wl.n_layers // 8)
        orc = OracleLayerSteps(wl, wl.max_ctx)
        times, keys = [], 0
        for i in range(args.warmup + args.steps):
            sec = 0.0
            for k in range(lps):
                j = i * lps + k
                layer, p = j % wl.n_layers, wl.prompt + j // wl.n_layers
                s_, _, k_ = orc.run_layer(layer, p)
                sec += s_
                if i >= args.warmup:
                    keys += k_
            if i >= args.warmup:
                times.append(sec)
        step_s = float(np.mean(times))
        v = wl.batch * lps / wl.n_layers / step_s
        sample = ("each step: the oracle over every (batch row, KV head) unit of %d of the %d "
                  "layers (%d units), layers in turn, positions advancing by one per %d steps; "
                  "%d keys over the %d timed steps; fp64 on %d threads (input generation "
                  "outside the clock)" % (lps, wl.n_layers, lps * orc.units_per_layer,
                                          wl.n_layers // lps, keys, args.steps, orc.cores))
        emit({"metric": metric, "value": v, "unit": "tokens/s", "n_gpus": args.gpus,
              "steps": args.steps, "warmup": args.warmup, "ms_per_step": step_s * 1e3,
              "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
              "data": "synthetic", "config": config, "impl": "reference",
              "step_fraction_of_decode_step": lps / wl.n_layers,
              "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": orc.cores,
                               "kind": "oracle", "sample": sample},
              "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                      "d2h_bytes_per_step": 0}})
        return

    if args.append_only:
        a = run_append(local, fp8=args.kv == "fp8", batch=args.batch)
        emit({"metric": "append GB/s", "value": a["gbs"], "unit": "GB/s", "n_gpus": 1,
              "higher_is_better": True, "dtype": "bf16", "data": "synthetic",
              "config": {"workload": a["workload"]}, "ms": a["ms"], "calls_timed": a["calls_timed"],
              "single_call_ms": a["single_call_ms"],
              "bytes_per_call": a["bytes_per_call"], "peak": hbm, "frac": a["gbs"] / hbm,
              "peak_source": peak_src})
        return
    if args.prefill_only:
        pre = run_prefill(args, local, fp8=args.kv == "fp8", workload=args.prefill_workload)
        emit({"metric": "prefill TFLOP/s", "value": pre["tflops"], "unit": "TFLOP/s",
              "n_gpus": 1, "higher_is_better": True,
              "dtype": "fp8-e4m3 KV" if args.kv == "fp8" else "bf16", "data": "synthetic",
              "config": {"workload": args.prefill_workload, "kv_format": args.kv}, "ms": pre["ms"],
              "flops": pre["flops"], "peak_tflops": tf_burst, "frac": pre["tflops"] / tf_burst,
              "frac_of_sustained": pre["tflops"] / tf_sust,
              "peak_source": peak_src})
        return
    r = run_gpu(args, wl, world, rank, local, fp8=args.kv == "fp8")
    r8 = None  # the same decode with the 8-bit cache format, as a secondary line
    if args.kv == "bf16" and not args.no_fp8 and wl.head_dim in (128, 256):
        a8 = argparse.Namespace(**vars(args))
        a8.steps, a8.e2e_steps = min(args.steps, 32), 2
        r8 = run_gpu(a8, wl, world, rank, local, fp8=True)
    pre = pre8 = pre256 = None
    if not args.no_prefill and rank == 0:
        pre = run_prefill(args, local)
        if not args.no_fp8:
            pre8 = run_prefill(args, local, fp8=True)
        pre256 = run_prefill(args, local, workload="single32k")
    app = run_append(local) if (not args.no_prefill and rank == 0) else None
    app8 = run_append(local, fp8=True) if (app is not None and not args.no_fp8) else None
    sec_lines = None
    if not args.no_secondary and args.kv == "bf16" and not (args.layers or args.batch):
        sec_lines = {}
        for name in SECONDARY_WORKLOADS:
            sec_lines[name] = run_secondary(args, name, world, rank, local, hbm)
    cal = None
    if rank == 0 and not args.no_calib:
        cal = run_calib(local)
    cb = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline and args.kv == "bf16":
        cb = cpu_baseline(wl, r["max_ctx"], r["t_first"] + 1)
    if rank != 0:
        return
    config["l2"] = ("each timed step preceded by a 2 x L2 read outside its events "
                    "(a layer-step reads less than 2 x L2)" if r["flush"] else
                    "inputs larger than L2 (each layer-step reads more than 2 x 129 MB of K/V)")
    line = {
        "metric": metric, "value": r["value"], "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": r["ms"] / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "fp8-e4m3 KV, f16 mma" if args.kv == "fp8" else "bf16",
        "data": "synthetic", "config": config,
        "hbm_gbs": r["step_bytes"] / (r["ms"] / args.steps * 1e-3) / 1e9,
        "roofline": {"bound": "hbm",
                     "kernel": "hwkv_decode_step (fused append + split kernel + combine), "
                               "layer 0 of each step",
                     "achieved": r["achieved_gbs"], "peak": hbm, "unit": "GB/s",
                     "frac": r["achieved_gbs"] / hbm, "peak_source": peak_src,
                     "frac_of_nominal_8tbs": r["achieved_gbs"] / NOMINAL_HBM_GBS,
                     "bytes_per_launch": r["bytes_avg"], "launch_ms": r["dec_avg_ms"],
                     "traffic": (r["bytes_avg"] * DECODE_TRAFFIC_PER_BYTE
                                 if DECODE_TRAFFIC_PER_BYTE else None),
                     "traffic_source": "ncu dram bytes of a 1-layer batch-2 capture, scaled by "
                                       "algorithmic bytes"},
        "residency_bytes": r["resid_bytes"],
        "positions": {"t_first_timed": r["t_first"], "t_end": r["t_end"],
                      "note": "tokens held per row before the first timed step and at the end "
                              "of the run (config.context is the workload's context)"},
        "e2e": {"value": r["e2e_value"], "unit": "tokens/s", "h2d_bytes_per_step": r["h2d"],
                "d2h_bytes_per_step": r["d2h"], "steps": r["e2e_steps"]},
        "gpu_launches": r["launches"],
        "clocks": r["clocks"],
        "graph_step": {"value": r["graph_value"], "unit": "tokens/s",
                       "ms_per_step": r["graph_ms"] / r["graph_steps"], "steps": r["graph_steps"],
                       "note": "the same step as one CUDA graph of %d hwkv_decode_step_graph "
                               "calls (lengths and tile plan on the device), replayed"
                               % wl.n_layers},
    }
    if r8 is not None:
        line["fp8_kv"] = {
            "value": r8["value"], "unit": "tokens/s", "ms_per_step": r8["ms"] / r8["steps"],
            "steps": r8["steps"], "decode_gbs": r8["achieved_gbs"], "frac": r8["achieved_gbs"] / hbm,
            "bytes_per_launch": r8["bytes_avg"], "graph_value": r8["graph_value"],
            "note": "same workload with the cache in E4M3 codes + one fp32 scale per row; "
                    "bytes counted as stored (codes and scales)"}
    if pre is not None:
        line["prefill"] = {"workload": "prefill64k", "tflops": pre["tflops"],
                           "peak_tflops": tf_burst, "frac": pre["tflops"] / tf_burst,
                           "peak_tflops_sustained": tf_sust,
                           "frac_of_sustained": pre["tflops"] / tf_sust,
                           "peak_source": peak_src, "ms": pre["ms"],
                           "tokens_per_s": pre["tokens_per_s"], "flops": pre["flops"]}
        tp = PREFILL_TENSOR_PIPE.get("prefill64k")
        if tp is not None:
            line["prefill"]["tensor_pipe_active_ncu"] = tp[0]
            line["prefill"]["tensor_pipe_source"] = tp[1]
        if pre8 is not None:
            line["prefill"]["fp8_kv"] = {
                "tflops": pre8["tflops"], "ms": pre8["ms"], "tokens_per_s": pre8["tokens_per_s"],
                "note": "same prompt with the cache in E4M3 codes + row scales; each call stages "
                        "q and the held/new K/V rows dequantized in fp16, then appends in 8 bits"}
        if pre256 is not None:
            line["prefill"]["head_dim_256"] = {
                "workload": "single32k", "tflops": pre256["tflops"],
                "frac": pre256["tflops"] / tf_burst, "ms": pre256["ms"],
                "tokens_per_s": pre256["tokens_per_s"], "flops": pre256["flops"],
                "note": "32K prompt in 8K chunks, batch 1, 24q/4kv, head_dim 256, windows "
                        "{full, 16384, 4096, 1024}"}
    if app is not None:
        line["append"] = {"workload": app["workload"], "gbs": app["gbs"], "frac": app["gbs"] / hbm,
                          "ms": app["ms"], "calls_timed": app["calls_timed"],
                          "single_call_ms": app["single_call_ms"],
                          "bytes_per_call": app["bytes_per_call"],
                          "note": "hwkv_append alone (the decode step fuses its one-token append); "
                                  "bytes = rows written + the same rows read; ms = the mean of "
                                  "consecutive calls timed together (single_call_ms: one call "
                                  "between its own events, the host's launch path inside)"}
        if app8 is not None:
            line["append"]["fp8_kv"] = {
                "gbs": app8["gbs"], "frac": app8["gbs"] / hbm, "ms": app8["ms"],
                "single_call_ms": app8["single_call_ms"],
                "bytes_per_call": app8["bytes_per_call"],
                "note": "8-bit cache: bf16 K/V read, E4M3 codes + fp32 row scales written"}
    if sec_lines is not None:
        line["other_workloads"] = sec_lines
    if cal is not None:
        line["seqcalib"] = cal
    if cb is not None:
        line["cpu_baseline"] = cb
    emit(line)


if __name__ == "__main__":
    main()
