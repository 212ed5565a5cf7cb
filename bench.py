#!/usr/bin/env python
"""Benchmark of AnchorKV decode attention on GB300.

Workload (default "70b-128k", the largest single-GPU configuration): Llama-3-70B
layer shape, 64 query / 8 KV heads (G = 8), head_dim 128, context 131072, batch 8,
2 % anchors and 10 % residual slots per side (about 20x smaller than the bf16
cache), a seeded compressed cache.  A step is one decode-attention call for one
layer with a fresh query set; the timed region cycles through 4 distinct layer
caches (874 MB, several times the 129 MB L2) and 64 fresh query sets, replayed
from CUDA graphs.  The metric is compressed bytes read per second (GB/s) and
microseconds per step.  Other workloads: "8b-32k" (GPU-encoded clustered K/V,
32 layers cycled), "8b-128k", and the ragged budget sweep "sweep-a<A>-r<R>".

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl akv|reference] [--workload NAME]

With --gpus N > 1 and no torch.distributed environment, the script starts N
ranks itself (torch.distributed.run on 127.0.0.1), one per GPU; each rank
encodes and decodes its own requests (data parallel by request, no collective
on the data path) and the line reports the whole job.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "decode-attn µs/step and HBM GB/s (% of ~8 TB/s) over 20× AnchorKV cache, 1 GB300"
WORKLOADS = {
    # name: (batch, n_kv_heads, n_q_heads, context, source)
    "8b-32k": (1, 8, 32, 32768, "encoded"),
    "8b-128k": (4, 8, 32, 131072, "seeded"),
    "70b-128k": (8, 8, 64, 131072, "seeded"),
}
# Budget and ragged-batch sweep at the 8B shape: 16 requests, contexts uniform in [8192, 131072]
# (one fixed draw), anchor fraction a % and residual-slot fraction r % per side.
SWEEP_BATCH = 16
SWEEP_POINTS = {f"sweep-a{a}-r{r}": (a / 100.0, r / 100.0) for a in (1, 2, 4) for r in (0, 5, 10, 20)}
for _name in SWEEP_POINTS:
    WORKLOADS[_name] = (SWEEP_BATCH, 8, 32, 0, "seeded")


def workload_lens(name: str, B: int, S: int) -> list:
    """Context length per request: S for the fixed workloads, the ragged draw for the sweep."""
    if name in SWEEP_POINTS:
        return [int(x) for x in np.random.default_rng(15).integers(8192, 131073, size=B)]
    return [S] * B


def workload_params(akv, name: str, **kw):
    """akv.Params of a workload (the sweep points set their budgets)."""
    fa, fr = SWEEP_POINTS.get(name, (0.02, 0.10))
    return akv.Params(anchor_frac=fa, res_frac_k=fr, res_frac_v=fr, **kw)
N_TOKENS = 64
# layer caches cycled per workload: enough distinct bytes to exceed the 129 MB L2 several times
DEFAULT_LAYERS = {"8b-32k": 32, "8b-128k": 8, "70b-128k": 4}
DEFAULT_LAYERS.update({n: 2 for n in SWEEP_POINTS})
# graph replays of (N_TOKENS x layers) steps timed by default, about ten seconds or less of device time
DEFAULT_REPLAYS = {"8b-32k": 100, "8b-128k": 40, "70b-128k": 40}
DEC_KERNEL_SRC = os.path.join(ROOT, "paper_2608_02901_gb300", "csrc", "akv_decode.cu")


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None)
    ap.add_argument("--warmup", type=int, default=None)
    ap.add_argument("--impl", default="akv", choices=["akv", "reference"])
    ap.add_argument("--workload", default="70b-128k", choices=sorted(WORKLOADS))
    ap.add_argument("--layers", type=int, default=None)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--codec", default="uniform", choices=["uniform", "lloyd"],
                    help="residual codec: 4 uniform levels on [min, max], or the Lloyd-Max codebook (AKV_FLAG_LLOYD)")
    ap.add_argument("--rope", action="store_true",
                    help="pre-RoPE keys with RoPE applied at decode (AKV_FLAG_ROPE, base 500000)")
    ap.add_argument("--suffix", type=int, default=0,
                    help="exact dense suffix: this many generated tokens per request, kept in bf16 and attended in "
                         "the same softmax (0 = none)")
    ap.add_argument("--launch-check", action="store_true",
                    help="start the ranks, have each report itself through the process group, print them and exit "
                         "(checks the N-rank launch; measures nothing)")
    ap.add_argument("--dense-context", action="store_true",
                    help="context only: torch scaled-dot-product attention decoding over the dense bf16 K/V of the same "
                         "shapes (a library kernel, not this repository's path)")
    args = ap.parse_args()
    if args.layers is None:
        args.layers = DEFAULT_LAYERS.get(args.workload, 2)
    chunk = N_TOKENS * args.layers
    if args.steps is None:
        args.steps = chunk * DEFAULT_REPLAYS.get(args.workload, 8)
    if args.warmup is None:
        args.warmup = chunk
    return args


TILE = 1024


def _tile_fixed(n):
    nw = (n + 63) // 64
    return 512 * nw + 16 * nw + 2 * ((2 * nw + 15) // 16 * 16)


def unit_bytes(S, k, nk, nv, G):
    """Compressed bytes one decode step reads for one (request, KV head), plus its q and out
    rows: anchors, tile table and tile blocks (record padding taken at its mean: 12 B of
    scale padding and 240 B of value-code group padding per tile; the benchmark itself
    reads the exact block sizes from the arena's tile tables)."""
    nt = (S + TILE - 1) // TILE
    fixed = sum(_tile_fixed(min(TILE, S - j * TILE)) for j in range(nt))
    return 512 * k + 4 * (2 * nt + 1) + fixed + 36 * (nk + nv) + 252 * nt + 2 * (2 * G * 128)


def arena_unit_bytes(torch, akv, p, lens, arena) -> list:
    """Exact bytes one decode reads from this arena per unit (anchors, tile table, the tile
    blocks as the table records them), plus the unit's q and out rows."""
    hdr = akv.akv_cache_header_host(p, lens)
    fixed = []
    offs = []
    for u in range(p.n_units):
        d = hdr[256 * (u + 1): 256 * (u + 2)]
        S, k, nt = int(d[0:4].view(np.int32)[0]), int(d[4:8].view(np.int32)[0]), int(d[16:20].view(np.int32)[0])
        o_tt = int(d[56:64].view(np.uint64)[0])
        offs.append(o_tt + 4 * nt)
        # (RoPE at decode: plus the stored tokens' positions)
        fixed.append(512 * k + 4 * (2 * nt + 1) + 2 * (2 * p.G * 128) + (4 * S if p.rope else 0))
    idx = torch.tensor([o + i for o in offs for i in range(4)], dtype=torch.long, device=arena.device)
    used = arena[idx].cpu().numpy().view(np.uint32).astype(np.int64)
    return [f + int(b) for f, b in zip(fixed, used)]


def arena_kernel_bytes(torch, akv, p, lens, arena):
    """Algorithmic bytes of each of the decode call's two launches over this arena: the score
    launch reads the anchor keys and the query rows (with RoPE at decode, the logits launch also
    the positions and key stream words); the decode launch the rest: anchor values, tile table,
    tile blocks, output rows (what the launches pass through the workspace is not counted)."""
    hdr = akv.akv_cache_header_host(p, lens)
    k_sum = sum(int(hdr[256 * (u + 1) + 4: 256 * (u + 1) + 8].view(np.int32)[0]) for u in range(p.n_units))
    s_sum = sum(int(hdr[256 * (u + 1): 256 * (u + 1) + 4].view(np.int32)[0]) for u in range(p.n_units))
    rows = p.n_units * 2 * p.G * 128
    total = arena_read_bytes(torch, akv, p, lens, arena)
    scores = 256 * k_sum + rows
    if p.rope:  # the RoPE logits launch also reads every token's position and key stream word
        scores += 8 * s_sum
    return scores, total - scores


def arena_read_bytes(torch, akv, p, lens, arena):
    """Exact bytes one decode reads from this arena, plus the q and out rows."""
    return sum(arena_unit_bytes(torch, akv, p, lens, arena))


def rank_seed(base: int, rank: int) -> int:
    """Seed of a rank's shard: every rank encodes and decodes its own batch (weak scaling)."""
    return base + 1000003 * rank


def free_port() -> int:
    import socket
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def launch_ranks(n: int) -> int:
    """Re-run this script as n ranks on one node (torch.distributed.run, rendezvous on 127.0.0.1);
    returns the launcher's exit code."""
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", f"--nproc-per-node={n}",
           "--master-addr=127.0.0.1", f"--master-port={free_port()}", os.path.abspath(__file__)] + sys.argv[1:]
    env = dict(os.environ, OMP_NUM_THREADS=os.environ.get("OMP_NUM_THREADS", "1"))
    return subprocess.run(cmd, env=env).returncode


def dist_setup(args):
    import torch
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args is not None and world != args.gpus:
        raise SystemExit(f"bench.py: --gpus {args.gpus} but the process group has WORLD_SIZE={world} ranks")
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        dist.init_process_group(backend=backend)
    if torch.cuda.is_available():
        torch.cuda.set_device(local)
    return rank, world, local


def dist_max(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device="cuda" if torch.cuda.is_available() else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def dist_barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        rows = []
        try:
            for line in open(self.path):
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        finally:
            os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"]}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower().startswith("active")})
        return {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


TRAFFIC_PROFILES = {"8b-32k": "akv_decode_8b32k_ncu.md", "8b-128k": "akv_decode_8b128k_ncu.md",
                    "70b-128k": "akv_decode_70b128k_ncu.md"}


def kernel_traffic(workload: str):
    """DRAM bytes per decode launch from the committed ncu summary of this workload, if there is one
    and it matches the current kernel source (the 128K captures cycle fewer layers than the benchmark;
    every launch reads one layer either way, so the bytes per launch are the same)."""
    src_hash = hashlib.sha256(open(DEC_KERNEL_SRC, "rb").read()).hexdigest()[:16]
    if workload not in TRAFFIC_PROFILES:
        return None
    path = os.path.join(ROOT, "profiles", TRAFFIC_PROFILES[workload])
    if not os.path.exists(path):
        return None
    vals = {}
    for line in open(path):
        if ":" in line and line.startswith("- "):
            key, val = line[2:].split(":", 1)
            vals[key.strip()] = val.strip().strip("`")
    if vals.get("kernel_source_sha256_16") != src_hash:
        return None
    try:
        return int(vals["dram_bytes_per_launch"])
    except (KeyError, ValueError):
        return None


def build_layers(torch, akv, gen, p, lens, layers, source, dev, rank=0):
    """Device arenas of `layers` distinct layer caches, the bytes one decode reads, and (GPU-encoded
    layers) the device time of the plain encoder per layer: CUDA events around each akv_encode call
    after one untimed encode, the layer's K/V already on the device."""
    arena_bytes, ws_bytes = akv.akv_cache_size(p, lens)
    shapes = akv.akv_unit_shapes(p, lens)
    arenas = []
    encode = None
    if source == "encoded":
        ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
        S = lens[0]
        times = []
        for layer in range(layers):
            K, V = gen.clustered_batch_torch(p.batch, p.n_kv_heads, S, seed=rank_seed(1000 + layer, rank), device=dev)
            arena = torch.empty(arena_bytes, dtype=torch.uint8, device=dev)
            if layer == 0:
                akv.akv_encode(p, lens, K, V, arena, ws)  # untimed: first-call set-up
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            akv.akv_encode(p, lens, K, V, arena, ws)
            e1.record()
            torch.cuda.synchronize()
            times.append(e0.elapsed_time(e1) * 1e3)
            arenas.append(arena)
            del K, V
        torch.cuda.synchronize()
        del ws
        us = sum(times) / len(times)
        tokens = p.batch * p.n_kv_heads * S
        encode = {"kernel_set": "akv_encode (plain encoder)", "us_per_layer": round(us, 2), "tokens": tokens,
                  "tokens_per_s": round(tokens / (us * 1e-6), 1),
                  "input_GB_per_s": round(tokens * 512 / (us * 1e-6) / 1e9, 1), "layers_timed": len(times)}
    else:
        base = None
        for layer in range(layers):
            if layer < 2:
                units = [akv.unit_host_from_logical(gen.seeded_cache(int(S), int(k), int(nk), int(nv), p.window,
                                                                       rank_seed(2000 + layer, rank), u))
                         for u, (S, k, nk, nv) in enumerate(shapes)]
                img = akv.akv_cache_pack_host(p, lens, units)
                arena = torch.from_numpy(img).to(dev)
                base = arena if layer == 0 else base
            else:  # further layers: device copies of the first two (distinct memory, same statistics)
                arena = arenas[layer % 2].clone()
            arenas.append(arena)
    # mean over the cycled layers of the exact bytes each decode reads
    step_bytes = sum(arena_read_bytes(torch, akv, p, lens, a) for a in arenas) / len(arenas)
    return arenas, arena_bytes, step_bytes, encode


def time_launches(torch, akv, step, n, stream, batch=32):
    """Mean device time of each of the decode call's two launches over n steps: an event before
    the call and the two the library records after its launches, on the launching stream.  Each
    batch of calls is queued behind a short device-side sleep, so that the calls run back to back
    on the device instead of waiting on the host between launches."""
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(n)]
    with torch.cuda.stream(stream):
        for trio in ev:  # creates the CUDA events the library records
            for e in trio:
                e.record(stream)
        stream.synchronize()
        try:
            for i0 in range(0, n, batch):
                torch.cuda._sleep(10_000_000)  # a few ms of device time while the host queues the batch
                for i in range(i0, min(n, i0 + batch)):
                    e0, e1, e2 = ev[i]
                    e0.record(stream)
                    akv.akv_decode_set_events(e1, e2)
                    step(i, stream)
        finally:
            akv.akv_decode_set_events()
        stream.synchronize()
    a = sum(e0.elapsed_time(e1) for e0, e1, _ in ev) * 1e3 / n
    b = sum(e1.elapsed_time(e2) for _, e1, e2 in ev) * 1e3 / n
    return a, b


def run_akv(args, rank, world, local):
    import torch

    import gen
    import paper_2608_02901_gb300 as akv

    dev = torch.device("cuda", local)
    B, H, Hq, S, source = WORKLOADS[args.workload]
    lens = workload_lens(args.workload, B, S)
    p = workload_params(akv, args.workload, batch=B, n_kv_heads=H, n_q_heads=Hq, seed=rank_seed(11, rank),
                        rot_seed=0x5EED, lloyd=args.codec == "lloyd", rope=args.rope)
    layers = args.layers
    arenas, arena_bytes, step_bytes, encode = build_layers(torch, akv, gen, p, lens, layers, source, dev, rank)
    n_tok = N_TOKENS
    qs = gen.queries_torch(n_tok * layers * B * Hq, seed=77 + rank, device=dev).view(n_tok, layers, B, Hq, 128)
    out = torch.empty((n_tok, layers, B, Hq, 128), dtype=torch.bfloat16, device=dev)
    chunk = n_tok * layers

    # the exact dense suffix of each layer (generated tokens in bf16), the same length for every request
    sfx = [None] * layers
    suffix_bytes = 0
    if args.suffix > 0:
        for layer in range(layers):
            kv = gen.queries_torch(2 * B * H * args.suffix, seed=5000 + 97 * layer + rank, device=dev)
            kv = kv.view(2, B, H, args.suffix, 128)
            sfx[layer] = akv.Suffix(kv[0].contiguous(), kv[1].contiguous(),
                                    torch.full((B,), args.suffix, dtype=torch.int32, device=dev))
        suffix_bytes = B * H * args.suffix * 2 * 256  # key and value rows, read by the suffix launch
        step_bytes += suffix_bytes

    # one decode workspace (anchor scores, partial sums) serves every call: they are stream-ordered
    dws = torch.empty(akv.akv_decode_workspace_size(p, lens, args.suffix), dtype=torch.uint8, device=dev)

    def step(i, stream=None):
        t, layer = divmod(i % chunk, layers)
        akv.akv_decode_attn(p, lens, arenas[layer], qs[t, layer], out[t, layer], None, 1.0, dws, stream,
                            suffix=sfx[layer])

    # warm-up (also sets kernel attributes before capture)
    for i in range(min(args.warmup, chunk)):
        step(i)
    torch.cuda.synchronize()
    stream = torch.cuda.Stream(device=dev)
    graphs = {}

    def graph_for(n):
        if n not in graphs:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                for i in range(n):
                    step(i, torch.cuda.current_stream())
            graphs[n] = g
        return graphs[n]

    full, rem = divmod(args.steps, chunk)
    g_full = graph_for(chunk) if full else None
    g_rem = graph_for(rem) if rem else None
    # graph warm-up: W steps total, at least 3
    w_left = max(3, args.warmup)
    with torch.cuda.stream(stream):
        while w_left > 0:
            graph_for(chunk).replay()
            w_left -= chunk
    torch.cuda.synchronize()

    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    dist_barrier(world)
    torch.cuda.synchronize()
    vis = os.environ.get("CUDA_VISIBLE_DEVICES", "")
    smi_index = vis.split(",")[local] if vis else str(local)
    with ClockSampler(smi_index) as clk:
        with torch.cuda.stream(stream):
            ev0.record(stream)
            for _ in range(full):
                g_full.replay()
            if g_rem is not None:
                g_rem.replay()
            ev1.record(stream)
        ev1.synchronize()
    torch.cuda.synchronize()
    dist_barrier(world)
    ms = ev0.elapsed_time(ev1)
    ms = dist_max(ms, world)
    clocks = clk.summary()
    sec = ms / 1e3
    # each launch of the step on its own, after the timed region (same layers, same order)
    us_scores, us_decode = time_launches(torch, akv, step, min(args.steps, max(chunk, 256)), stream)
    kb = [arena_kernel_bytes(torch, akv, p, lens, a) for a in arenas]
    scores_bytes = sum(b[0] for b in kb) / len(kb) + suffix_bytes
    decode_bytes = sum(b[1] for b in kb) / len(kb)
    value = world * step_bytes * args.steps / sec / 1e9
    us_step = ms * 1e3 / args.steps

    # End to end through the C ABI with host buffers: every step copies its query set in from
    # pinned host memory, decodes, copies the output back to pinned host memory and waits for
    # it on the host.  The three operations of a step are replayed from one CUDA graph (the
    # way a serving loop issues them); the same steps issued eagerly from Python are reported
    # beside it.
    e2e_steps = min(args.steps, chunk, 64)
    q_host = torch.empty((e2e_steps, B, Hq, 128), dtype=torch.bfloat16, pin_memory=True)
    for i in range(e2e_steps):
        t, layer = divmod(i, layers)
        q_host[i].copy_(qs[t, layer].cpu())
    o_host = torch.empty((e2e_steps, B, Hq, 128), dtype=torch.bfloat16, pin_memory=True)
    q_dev = torch.empty((B, Hq, 128), dtype=torch.bfloat16, device=dev)
    o_dev = torch.empty((B, Hq, 128), dtype=torch.bfloat16, device=dev)

    def e2e_ops(i, s):
        q_dev.copy_(q_host[i], non_blocking=True)
        akv.akv_decode_attn(p, lens, arenas[i % layers], q_dev, o_dev, None, 1.0, dws, s, suffix=sfx[i % layers])
        o_host[i].copy_(o_dev, non_blocking=True)

    e2e_graphs = []
    for i in range(e2e_steps):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            e2e_ops(i, torch.cuda.current_stream())
        e2e_graphs.append(g)
    with torch.cuda.stream(stream):  # replays run on the current stream: make it the one waited on
        for g in e2e_graphs:  # warm-up
            g.replay()
        stream.synchronize()
    dist_barrier(world)
    with torch.cuda.stream(stream):
        t0 = time.perf_counter()
        for g in e2e_graphs:
            g.replay()
            stream.synchronize()
        e2e_sec = dist_max(time.perf_counter() - t0, world)
    with torch.cuda.stream(stream):
        t0 = time.perf_counter()
        for i in range(e2e_steps):
            e2e_ops(i, stream)
            stream.synchronize()
        eager_sec = dist_max(time.perf_counter() - t0, world)
    h2d = B * Hq * 128 * 2
    e2e = {"value": round(world * step_bytes * e2e_steps / e2e_sec / 1e9, 3), "unit": "GB/s",
           "us_per_step": round(e2e_sec * 1e6 / e2e_steps, 3), "steps": e2e_steps,
           "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": h2d,
           "how": "per step: H2D copy of the query set from pinned memory, akv_decode_attn, D2H copy of the output "
                  "to pinned memory (one CUDA graph per step), host synchronisation",
           "eager_us_per_step": round(eager_sec * 1e6 / e2e_steps, 3)}

    peaks = {}
    try:
        peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except (OSError, ValueError):
        pass
    peak = float(peaks.get("hbm_gbs", 6800.0))
    # the dominant kernel (the decode launch): its algorithmic bytes over its mean launch time
    achieved = decode_bytes / (us_decode * 1e-6) / 1e9
    roofline = {"bound": "hbm", "achieved": round(achieved, 2), "peak": peak, "unit": "GB/s",
                "frac": round(achieved / peak, 4), "traffic": kernel_traffic(args.workload),
                "kernel": "akv_decode_kernel", "launch_us": round(us_decode, 3),
                "bytes_per_launch": round(decode_bytes),
                "peak_source": "measured" if "hbm_gbs" in peaks else "fallback",
                "frac_of_8tbs": round(achieved / 8000.0, 4),
                "step": {"bytes": round(step_bytes), "achieved": round(step_bytes / (sec / args.steps) / 1e9, 2),
                         "frac": round(step_bytes / (sec / args.steps) / 1e9 / peak, 4)},
                "scores_kernel": {"kernel": ("akv_rope_logits_kernel" if args.rope else "akv_scores_tc_kernel")
                                  + (" + akv_suffix_kernel" if args.suffix > 0 else ""),
                                  "launch_us": round(us_scores, 3),
                                  "bytes_per_launch": round(scores_bytes),
                                  "achieved": round(scores_bytes / (us_scores * 1e-6) / 1e9, 2)},
                "launch_timing": "steps after the timed region, queued in batches behind a device sleep so that "
                                 "they run back to back: an event before each call and the two the library records "
                                 "after its launches (akv_decode_set_events)"}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(torch, akv, p, lens, arenas[0], encoded=source == "encoded")

    line = {
        "metric": METRIC, "value": round(value, 3), "unit": "GB/s", "us_per_step": round(us_step, 4),
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms / args.steps, 6),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (seeded clustered K/V, encoded on GPU)" if source == "encoded" else "synthetic (seeded cache)",
        "config": {"workload": args.workload, "batch": B, "n_kv_heads": H, "n_q_heads": Hq,
                   "context": S if args.workload not in SWEEP_POINTS else f"ragged U[8192, 131072]: {lens}",
                   "anchor_frac": p.anchor_frac, "res_frac": p.res_frac_k, "layers_cycled": layers,
                   "suffix_tokens": args.suffix, "codec": args.codec, "rope_at_decode": args.rope,
                   "fresh_queries": N_TOKENS, "arena_bytes_per_layer": arena_bytes,
                   "l2": f"inputs larger than L2: {layers} distinct layer caches, {layers * arena_bytes / 1e6:.0f} MB cycled",
                   "timing": "CUDA graph replay, CUDA events on the launching stream", "parallelism": f"dp{world}"},
        "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": (3 if args.suffix > 0 else 2) * args.steps, "clocks": clocks,
    }
    if encode is not None:  # context: the compression pass of the layers this run decodes
        line["encode"] = encode
    if rank == 0:
        print(json.dumps(line), flush=True)


def _oracle_units_from_arena(torch, arena):
    import oracle
    return oracle.unpack_arena(arena.cpu().numpy())


def cpu_baseline(torch, akv, p, lens, arena, budget_s=16.0, encoded=False):
    """The fp64 oracle, as it stands, on the host cores, over the same layer cache the GPU reads:
    whole layer steps with OpenMP over the units (threads = min(cores, units)), then single units
    on one core.  Bytes are the exact bytes of the units attended (the tile tables' sizes).  For a
    GPU-encoded workload also the oracle's encode of one unit of the same shape on one core."""
    import gen
    import oracle
    units = _oracle_units_from_arena(torch, arena)
    ub = arena_unit_bytes(torch, akv, p, lens, arena)
    G, n = p.G, p.n_units
    q = gen.queries(n * G, seed=5).reshape(n, G, 128)
    nproc = os.cpu_count() or 1
    threads = min(nproc, n)
    done, t0 = 0, time.perf_counter()
    while True:
        oracle.attend(units, q, G, 1.0, p.rot_seed)
        done += 1
        if time.perf_counter() - t0 > budget_s / 2:
            break
    sec = time.perf_counter() - t0
    one, b1, t1 = 0, 0, time.perf_counter()
    sel = np.zeros(n, np.uint8)
    while True:
        sel[:] = 0
        sel[one % n] = 1
        oracle.attend(units, q, G, 1.0, p.rot_seed, sel=sel)
        b1 += ub[one % n]
        one += 1
        if time.perf_counter() - t1 > budget_s / 2:
            break
    sec1 = time.perf_counter() - t1
    enc = None
    if encoded:  # the compression pass: one unit of the workload's shape, clustered K/V, one core
        S = int(lens[0])
        K, V = gen.clustered_batch(1, 1, [S], seed=1000)
        t2 = time.perf_counter()
        oracle.encode(K, V, [S], 1, p.anchor_frac, p.res_frac_k, p.res_frac_v, p.window, p.seed, p.rot_seed,
                      rotate=p.rotate, lloyd=p.lloyd)
        sec2 = time.perf_counter() - t2
        enc = {"kind": "oracle encode", "cores": 1, "tokens": S, "seconds": round(sec2, 3),
               "tokens_per_s": round(S / sec2, 1), "sample": f"one unit of {S} tokens"}
    out = {"value": round(sum(ub) * done / sec / 1e9, 5), "unit": "GB/s", "cores": threads, "nproc": nproc,
            "kind": "oracle",
            "sample": f"{done} full layer steps of the workload's first layer cache ({n} units, OpenMP over units)",
            "seconds": round(sec, 2), "us_per_step": round(sec * 1e6 / done, 1),
            "single_core": {"value": round(b1 / sec1 / 1e9, 5), "unit": "GB/s", "cores": 1,
                            "sample": f"{one} single units of the same layer, one at a time", "seconds": round(sec1, 2)}}
    if enc is not None:
        out["encode"] = enc
    return out


def run_reference(args, rank, world, local):
    """The oracle (fp64 CPU) timed as the reference arm on a bounded sample of the same workload."""
    if rank != 0:
        return
    import gen
    import oracle
    import paper_2608_02901_gb300 as akv_params_only  # Params/shape helpers are pure host code
    B, H, Hq, S, source = WORKLOADS[args.workload]
    S = max(workload_lens(args.workload, B, S))  # the longest request of a ragged batch
    G = Hq // H
    p = workload_params(akv_params_only, args.workload, batch=1, n_kv_heads=1, n_q_heads=G, seed=11, rot_seed=0x5EED)
    # one (request, KV head) unit of the workload; each step attends one query group over a prefix of it
    k, nk, nv = oracle.unit_shape(S, p.anchor_frac, p.res_frac_k, p.res_frac_v, p.window)
    if source == "encoded":
        K, V = gen.clustered_batch(1, 1, [S], seed=1000)
        unit = oracle.encode(K, V, [S], 1, p.anchor_frac, p.res_frac_k, p.res_frac_v, p.window, p.seed,
                             p.rot_seed)[0]
    else:
        d = gen.seeded_cache(S, k, nk, nv, p.window, 2000, 0)
        unit = oracle.alloc_unit(S, k, nk, nv)
        for f in ("anchor_k", "anchor_v", "anchor_pos", "idx_k", "gam_k", "idx_v", "gam_v", "res_k", "codes_k",
                  "scale_k", "min_k", "res_v", "codes_v", "scale_v", "min_v"):
            getattr(unit, f)[...] = d[f]
    total_budget = 150.0
    per_step = total_budget / max(1, args.steps + args.warmup)
    # estimate the oracle's time per position on this host
    q = gen.queries(G, seed=3)
    t0 = time.perf_counter()
    oracle.attend([unit], q.reshape(1, G, 128), G, 1.0, p.rot_seed)
    per_pos = (time.perf_counter() - t0) / S
    P = int(max(64, min(S, per_step / max(per_pos, 1e-12))))
    sub = _prefix_unit(oracle, unit, P)
    sub_bytes = unit_bytes(sub.S, sub.k, sub.nk, sub.nv, G)
    for _ in range(args.warmup):
        oracle.attend([sub], q.reshape(1, G, 128), G, 1.0, p.rot_seed)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle.attend([sub], q.reshape(1, G, 128), G, 1.0, p.rot_seed)
    sec = time.perf_counter() - t0
    val = sub_bytes * args.steps / sec / 1e9
    line = {"impl": "reference", "metric": METRIC, "value": round(val, 6), "unit": "GB/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(sec * 1e3 / args.steps, 6),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": args.workload, "context": S, "sample_positions": P},
            "cpu_baseline": {"value": round(val, 6), "unit": "GB/s", "cores": 1, "kind": "oracle",
                             "sample": f"one query group over the first {P} of {S} positions of one unit per step"},
            "e2e": {"value": round(val, 6), "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def _prefix_unit(oracle, u, P):
    """The first P positions of a unit's logical cache (all anchors kept, residual slots restricted)."""
    if P >= u.S:
        return u
    mk, mv = u.res_k < P, u.res_v < P
    sub = oracle.alloc_unit(P, u.k, int(mk.sum()), int(mv.sum()))
    sub.anchor_k[...] = u.anchor_k
    sub.anchor_v[...] = u.anchor_v
    sub.anchor_pos[...] = u.anchor_pos
    for f in ("idx_k", "gam_k", "idx_v", "gam_v"):
        getattr(sub, f)[...] = getattr(u, f)[:P]
    sub.res_k[...] = u.res_k[mk]
    sub.codes_k[...] = u.codes_k[mk]
    sub.scale_k[...] = u.scale_k[mk]
    sub.min_k[...] = u.min_k[mk]
    sub.res_v[...] = u.res_v[mv]
    sub.codes_v[...] = u.codes_v[mv]
    sub.scale_v[...] = u.scale_v[mv]
    sub.min_v[...] = u.min_v[mv]
    return sub


def run_dense_context(args, rank, world, local):
    """Dense bf16 decode attention over the uncompressed K/V of the workload's shapes, timed the way
    the main line is (CUDA graph, events, inputs larger than L2): the cost the compressed cache is
    compared against.  Random data: only the time is of interest."""
    import torch
    import torch.nn.functional as F
    if rank != 0:
        return
    dev = torch.device("cuda", local)
    B, H, Hq, S, _ = WORKLOADS[args.workload]
    lens = workload_lens(args.workload, B, S)
    Smax = max(lens)
    per_layer = 2 * B * H * Smax * 128 * 2
    layers = max(1, min(args.layers, int(math.ceil(400e6 / per_layer))))  # > 3x L2 in total
    g = torch.Generator(device=dev)
    g.manual_seed(5)
    Ks = [torch.randn((B, H, Smax, 128), generator=g, device=dev, dtype=torch.bfloat16) for _ in range(layers)]
    Vs = [torch.randn((B, H, Smax, 128), generator=g, device=dev, dtype=torch.bfloat16) for _ in range(layers)]
    q = torch.randn((B, Hq, 1, 128), generator=g, device=dev, dtype=torch.bfloat16) / math.sqrt(128)
    mask = None
    if len(set(lens)) > 1:  # ragged batch: positions past a request's length masked out
        pos = torch.arange(Smax, device=dev)
        mask = (pos[None, None, None, :] < torch.tensor(lens, device=dev)[:, None, None, None])
    outs = torch.empty((B, Hq, 1, 128), device=dev, dtype=torch.bfloat16)

    def step(i):
        outs.copy_(F.scaled_dot_product_attention(q, Ks[i % layers], Vs[i % layers], attn_mask=mask, scale=1.0,
                                                  enable_gqa=True))

    for i in range(max(3, layers)):
        step(i)
    torch.cuda.synchronize()
    stream = torch.cuda.Stream(device=dev)
    n = max(layers, 64)
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        for i in range(n):
            step(i)
    graph.replay()
    torch.cuda.synchronize()
    reps = max(1, args.steps // n)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record()
        for _ in range(reps):
            graph.replay()
        e1.record()
    torch.cuda.synchronize()
    us = e0.elapsed_time(e1) * 1e3 / (reps * n)
    dense_bytes = sum(2 * H * L * 128 * 2 for L in lens)
    print(json.dumps({"impl": "dense-sdpa-context", "workload": args.workload, "us_per_step": round(us, 3),
                      "dense_bytes_per_step": dense_bytes, "GB/s": round(dense_bytes / (us * 1e-6) / 1e9, 1),
                      "layers_cycled": layers, "note": "torch scaled_dot_product_attention on dense bf16 K/V "
                      "(library kernel, context only)"}), flush=True)


def run_launch_check(args, rank, world, local):
    """Every rank reports (rank, local rank, world size) through the process group; rank 0 prints them."""
    import torch
    if world > 1:
        import torch.distributed as dist
        mine = [rank, local, world, os.getpid()]
        got = [None] * world
        dist.all_gather_object(got, mine)
    else:
        got = [[rank, local, world, os.getpid()]]
    if rank == 0:
        print(json.dumps({"launch_check": True, "n_gpus": args.gpus, "world_size": world,
                          "ranks": sorted(g[0] for g in got), "local_ranks": sorted(g[1] for g in got),
                          "distinct_processes": len({g[3] for g in got}),
                          "backend": "nccl" if torch.cuda.is_available() else "gloo"}), flush=True)


def main():
    args = parse()
    if args.gpus > 1 and "WORLD_SIZE" not in os.environ:
        sys.exit(launch_ranks(args.gpus))
    rank, world, local = dist_setup(args)
    try:
        if args.launch_check:
            run_launch_check(args, rank, world, local)
        elif args.dense_context:
            run_dense_context(args, rank, world, local)
        elif args.impl == "reference":
            run_reference(args, rank, world, local)
        else:
            run_akv(args, rank, world, local)
    finally:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
