#!/usr/bin/env python
"""Verified tokens/s of DiP-SD batch verification on one GB300 (and per-stage HBM roofline).

One step = one pipeline stage verified end to end on the GPU through the C ABI
(dipsd_verify_batch: verify attention over every user's paged KV cache, then
speculative sampling over the vocabulary) on the Qwen3-32B-shaped batch
(B=8, L_i ~ U{1..8}, context 1024, 64/8/128 heads, V=151936).  Inputs are
resident in HBM; consecutive steps rotate over enough device copies of the
batch that their inputs exceed L2, so every step reads cold data; the K calls
are captured in one CUDA graph, and the graph is replayed back to back until
at least --min-replay-ms of device time has run, each replay of exactly K
steps between a pair of CUDA events: the value is the median replay, with the
spread beside it.  The line also carries:
  * e2e: the same steps through the Python API as plain calls (the library's
    host validation and planning included), each step copying its inputs from
    pinned host memory and its results back; e2e_graph: the same calls
    captured as one CUDA graph;
  * per-stage roofline figures against the measured HBM copy bandwidth, on
    this workload and (--extra 1, the default) on workloads 3 and 4, and the
    sustained rate of workload 5's pipelined schedule;
  * the clocks seen while timing, and the fp64 CPU oracle on the host cores.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl dipsd|reference]
Under torchrun (N > 1) every rank verifies its own replica of the batch.
"""
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

L2_FLUSH_BYTES = 256 << 20
L2_BYTES = 126 << 20
FALLBACK_HBM_GBS = 6800.0


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["dipsd", "reference"], default="dipsd")
    ap.add_argument("--workload", type=int, default=2, help="workload id (2 = the headline batch)")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--cpu-seconds", type=float, default=10.0,
                    help="budget of the CPU oracle baseline (0: skip it, for the large non-headline workloads)")
    ap.add_argument("--min-replay-ms", type=float, default=300.0,
                    help="device time each timed graph is replayed for (at least 3 replays)")
    ap.add_argument("--extra", type=int, default=1,
                    help="1: also time workloads 3 and 4 per stage and workload 5's pipelined schedule")
    return ap.parse_args()


def workload_config(b, wl, seed):
    from workloads import CONFIG_NAMES
    return {"workload": CONFIG_NAMES[wl], "B": int(b.B), "L": [int(x) for x in b.L],
            "ctx": [int(x) for x in b.ctx], "heads": f"{b.Hq}/{b.Hkv}/{b.D}", "V": int(b.V),
            "page": 16, "seed": seed}


def step_bytes(b):
    return attention_bytes(b) + spec_bytes(b)


def copies_for(b):
    """Device copies of a batch that consecutive steps rotate over: their
    inputs together exceed L2 twice over, so every step reads cold data."""
    return max(2, math.ceil(2 * L2_BYTES / step_bytes(b)))


def bench_config(b, wl, seed, world):
    """`config` of the bench line, the same in both arms."""
    cfg = workload_config(b, wl, seed)
    R = copies_for(b)
    cfg["l2"] = (f"inputs rotated over {R} device copies ({R * step_bytes(b) / 1e6:.0f} MB > 2 x L2), "
                 "K steps back to back as one CUDA graph replay")
    cfg["parallelism"] = "replicas" if world > 1 else "single"
    return cfg


def read_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            pk = json.load(f)
        return float(pk["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples while the timed loops run."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-f", self.path], stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        time.sleep(0.2)
        self.proc.terminate()
        self.proc.wait(timeout=10)
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[k] for r in rows for k in range(4) if r[5 + k].lower() == "active"})
        return {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows),
                "power_w_max": max((float(r[3]) for r in rows if r[3].replace(".", "").isdigit()), default=None)}


def attention_bytes(b):
    """Algorithmic HBM bytes of one verify-attention launch: each user's K and V rows
    (kv_len x Hkv x D x 2 B, twice), the Q read and the output write."""
    kv = int(b.kv_len.sum()) * b.Hkv * b.D * 2 * 2
    return kv + 2 * b.sum_T * b.Hq * b.D * 2


def spec_bytes(b):
    """Algorithmic HBM bytes of one spec-verify launch: one pass over every target-logit
    row and every draft-logit row (the resample re-read is implementation overhead)."""
    el = 2 if b.logit_dtype == "bf16" else 4
    return (b.sum_T + b.sum_L) * b.V * el


def sparse_bytes(b, K=64):
    """Algorithmic bytes of one sparse-payload launch: one pass over every
    target-logit row, plus the table (K entries of 8 bytes) and log q(d) per draft row."""
    el = 2 if b.logit_dtype == "bf16" else 4
    return b.sum_T * b.V * el + b.sum_L * (8 * K + 4)


def source_hash(paths):
    """Hash of the kernel sources with comments and blank lines removed, so a
    traffic record follows the code, not its commentary."""
    import re
    h = hashlib.sha256()
    for p in paths:
        with open(os.path.join(ROOT, p)) as f:
            text = f.read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        text = re.sub(r"//[^\n]*", "", text)
        h.update("\n".join(line.rstrip() for line in text.splitlines() if line.strip()).encode())
    return h.hexdigest()[:16]


def recorded_traffic(kernel, workload, src_hash):
    """DRAM bytes (read + write) per launch from the committed ncu summary, if
    one was taken of this kernel on this workload and this source."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f).get(f"{kernel}@workload{workload}")
    except (OSError, ValueError):
        return None
    if not rec or rec.get("source_hash") != src_hash:
        return None
    return rec.get("dram_bytes_per_launch")


def oracle_step(b_host, users):
    """Oracle on the chosen users of the batch; returns the tokens it emitted."""
    import oracle
    from workloads import offsets
    users = np.asarray(users)
    qo, lo = offsets(b_host["T"]), offsets(b_host["L"])
    rows = np.concatenate([np.arange(qo[i], qo[i + 1]) for i in users])
    drows = np.concatenate([np.arange(lo[i], lo[i + 1]) for i in users] + [np.zeros(0, int)])
    oracle.verify_attention(b_host["q"][rows], b_host["k"], b_host["v"], b_host["bt"][users],
                            b_host["ctx"][users], b_host["L"][users], b_host["scale"])
    r = oracle.spec_verify(b_host["L"][users], b_host["z"][rows], b_host["w"][drows], b_host["d"][drows],
                           b_host["u"][rows])
    return int(r["out_offsets"][-1])


def host_copy(b):
    return {"q": b.q.double().cpu().numpy(), "k": b.k_cache.double().cpu().numpy(),
            "v": b.v_cache.double().cpu().numpy(), "bt": b.block_table.cpu().numpy(),
            "ctx": b.ctx, "L": b.L, "T": b.T, "scale": b.scale,
            "z": b.target_logits.double().cpu().numpy(), "w": b.draft_logits.double().cpu().numpy(),
            "d": b.draft_tokens.cpu().numpy(), "u": b.uniforms.cpu().numpy()}


def cpu_baseline(b, budget_s):
    """The oracle as it stands on the host cores: whole batches until the budget is spent."""
    hb = host_copy(b)
    users = list(range(b.B))
    t0 = time.perf_counter()
    tokens, reps = 0, 0
    while True:
        tokens += oracle_step(hb, users)
        reps += 1
        if time.perf_counter() - t0 >= budget_s:
            break
    dt = time.perf_counter() - t0
    return {"value": tokens / dt, "unit": "verified tokens/s", "cores": os.cpu_count(), "kind": "oracle",
            "sample": f"{reps} full batch(es) of the workload ({b.B} users), fp64 numpy, {dt:.1f} s",
            "threads": "numpy/BLAS defaults"}


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if rank != 0:
        return
    from workloads import make_config
    b = make_config(args.workload, seed=args.seed, device="cpu")
    hb = host_copy(b)
    users = list(range(b.B))
    for _ in range(args.warmup):
        oracle_step(hb, users)
    t0 = time.perf_counter()
    tokens = 0
    for _ in range(args.steps):
        tokens += oracle_step(hb, users)
    dt = time.perf_counter() - t0
    value = tokens / dt
    line = {"metric": "verified tokens/s (one verification stage: attention + speculative sampling)",
            "value": value, "unit": "verified tokens/s", "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1000 * dt / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": bench_config(b, args.workload, args.seed, world), "impl": "reference",
            "cpu_baseline": {"value": value, "unit": "verified tokens/s", "cores": os.cpu_count(),
                             "kind": "oracle", "sample": f"{args.steps} full batch(es) of the workload"},
            "e2e": {"value": value, "unit": "verified tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------- timing
def packed_layout(tensors, align=256):
    """One uint8 buffer holding the tensors back to back (each at a 256-byte
    aligned offset), and a function that returns their views into any buffer
    of that layout."""
    import torch
    offs, n = [], 0
    for t in tensors:
        offs.append(n)
        n += -(-(t.numel() * t.element_size()) // align) * align
    buf = torch.zeros(n, dtype=torch.uint8)
    for t, o in zip(tensors, offs):
        buf[o:o + t.numel() * t.element_size()].copy_(t.contiguous().view(-1).view(torch.uint8))

    def views_of(x):
        return [x[o:o + t.numel() * t.element_size()].view(t.dtype).view(t.shape) for t, o in zip(tensors, offs)]
    return buf, views_of


def capture(fn, n, R, stream):
    """A CUDA graph of n consecutive calls fn(0), .., fn(n - 1) (lazy set-up
    settled outside the capture) and the library kernels one replay launches."""
    import torch
    from paper_2604_20919_gb300 import dipsd
    g = torch.cuda.CUDAGraph()
    side = torch.cuda.Stream()
    side.wait_stream(stream)
    with torch.cuda.stream(side):
        for i in range(R):
            fn(i)
    stream.wait_stream(side)
    torch.cuda.synchronize()
    n0 = dipsd.dipsd_launch_count()
    # captured on the stream that made the warm-up calls: the library's
    # per-stream resources (verify_batch's second stream) exist by then
    with torch.cuda.graph(g, stream=side):
        for i in range(n):
            fn(i)
    torch.cuda.synchronize()
    return g, dipsd.dipsd_launch_count() - n0


def replay_ms(g, stream, reps, barrier=None):
    """reps replays of a graph, each between a pair of CUDA events on the
    launching stream (synchronised on both sides): ms per replay."""
    import torch
    out = []
    for _ in range(reps):
        if barrier:
            barrier()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        g.replay()
        e1.record(stream)
        torch.cuda.synchronize()
        out.append(e0.elapsed_time(e1))
    return out


def replay_stats(g, n, stream, min_ms):
    """ms per call of an n-call graph: median, min and max over replays run
    until min_ms of device time (at least 3 replays)."""
    first = replay_ms(g, stream, 2)[1]
    reps = max(3, min(2000, math.ceil(min_ms / max(first, 1e-3))))
    t = np.asarray(replay_ms(g, stream, reps)) / n
    return {"ms": float(np.median(t)), "ms_min": float(t.min()), "ms_max": float(t.max()), "replays": reps,
            "calls_per_replay": n}


def stage_entry(st, alg_bytes, hbm_peak):
    gbs = alg_bytes / st["ms"] / 1e6
    return dict(st, alg_bytes=alg_bytes, gbs=gbs, frac_of_measured_hbm=gbs / hbm_peak, frac_of_8000=gbs / 8000.0)


def device_batch(b, dev, R):
    """R device copies of a batch's per-step inputs (the KV cache cloned too)."""
    copies = []
    for k in range(R):
        kc = b.k_cache if k == 0 else b.k_cache.clone()
        vc = b.v_cache if k == 0 else b.v_cache.clone()
        copies.append(dict(q=b.q.to(dev), z=b.target_logits.to(dev), w=b.draft_logits.to(dev),
                           d=b.draft_tokens.to(dev), kc=kc, vc=vc))
    return copies


def measure_workload(wl, args, dev, stream, hbm_peak):
    """Per-stage times of one workload (attention alone, speculative sampling
    alone, the whole verify_batch step), inputs rotated over device copies
    larger than L2 twice over."""
    import torch
    from paper_2604_20919_gb300 import dipsd
    from workloads import CONFIG_NAMES, make_config
    b = make_config(wl, seed=args.seed, device="cpu", kv_device=dev)
    R = copies_for(b)
    copies = device_batch(b, dev, R)
    bt = b.block_table.to(dev)
    attn_out = torch.empty_like(copies[0]["q"])
    outs = dipsd.spec_outputs(b.L, dev)
    ws = dipsd.workspace(dipsd.dipsd_verify_batch_workspace_size(b.members, b.L, b.ctx, b.Hq, b.Hkv, b.D, b.V), dev)

    def step(k):
        c = copies[k % R]
        dipsd.dipsd_verify_batch(b.members, b.L, b.ctx, c["q"], c["kc"], c["vc"], bt, b.scale, c["z"], c["w"],
                                 c["d"], b.seed, attn_out=attn_out, outputs=outs, ws=ws)

    def attn_only(k):
        c = copies[k % R]
        dipsd.dipsd_verify_attention(b.L, b.ctx, c["q"], c["kc"], c["vc"], bt, b.scale, out=attn_out, ws=ws)

    def spec_only(k):
        c = copies[k % R]
        dipsd.dipsd_spec_verify(b.L, b.members, b.seed, c["z"], c["w"], c["d"], outputs=outs, ws=ws)

    for i in range(3):
        step(i)
    torch.cuda.synchronize()
    # about 20 ms of device time per replay
    n = int(min(500, max(5, 0.02 / (step_bytes(b) / 4.0e12))))
    res = {"workload": CONFIG_NAMES[wl], "B": int(b.B), "sum_T": int(b.sum_T)}
    for name, fn, by in (("step", step, step_bytes(b)), ("verify_attention", attn_only, attention_bytes(b)),
                         ("spec_verify", spec_only, spec_bytes(b))):
        g, _ = capture(fn, n, R, stream)
        res[name] = stage_entry(replay_stats(g, n, stream, args.min_replay_ms), by, hbm_peak)
        del g
    emitted = int(outs[1][-1].item())
    res["step"]["verified_tokens_per_s"] = emitted / (res["step"]["ms"] / 1000.0)
    res["emitted_tokens_per_step"] = emitted
    res["l2"] = f"inputs rotated over {R} device copies ({R * step_bytes(b) / 1e6:.0f} MB)"
    assert dipsd.device_status(ws) == 0
    del copies, attn_out, outs, ws, bt
    torch.cuda.empty_cache()
    return res


def run_dipsd(args):
    import torch
    import torch.distributed as dist
    from paper_2604_20919_gb300 import dipsd
    from workloads import make_config

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    barrier = dist.barrier if world > 1 else None
    dipsd.load()
    hbm_peak, peak_kind = read_peaks()

    # each rank verifies its own replica (independent users): weak scaling, no collective
    b = make_config(args.workload, seed=args.seed + rank, device="cpu", kv_device=dev)
    R = copies_for(b)
    copies = device_batch(b, dev, R)
    bt = b.block_table.to(dev)
    attn_out = torch.empty_like(copies[0]["q"])
    outs = dipsd.spec_outputs(b.L, dev)
    ws = dipsd.workspace(dipsd.dipsd_verify_batch_workspace_size(b.members, b.L, b.ctx, b.Hq, b.Hkv, b.D, b.V), dev)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    def step(k):
        c = copies[k % R]
        dipsd.dipsd_verify_batch(b.members, b.L, b.ctx, c["q"], c["kc"], c["vc"], bt, b.scale, c["z"], c["w"],
                                 c["d"], b.seed, attn_out=attn_out, outputs=outs, ws=ws)

    def attn_only(k):
        c = copies[k % R]
        dipsd.dipsd_verify_attention(b.L, b.ctx, c["q"], c["kc"], c["vc"], bt, b.scale, out=attn_out, ws=ws)

    def spec_only(k):
        c = copies[k % R]
        dipsd.dipsd_spec_verify(b.L, b.members, b.seed, c["z"], c["w"], c["d"], outputs=outs, ws=ws)

    # the verify tokens' own K/V rows (already in the cache), for the append path
    bt_h = b.block_table.numpy()
    pos = [(i, int(b.ctx[i]) + t) for i in range(b.B) for t in range(int(b.L[i]) + 1)]
    blk = torch.tensor([int(bt_h[i, p // 16]) for i, p in pos], device=dev)
    slot = torch.tensor([p % 16 for _, p in pos], device=dev)
    new_k = b.k_cache[blk, :, slot].contiguous()
    new_v = b.v_cache[blk, :, slot].contiguous()

    # sparse draft payload of the same batch (K = 64 table entries per draft row)
    from workloads import make_sparse_draft
    sdraft = make_sparse_draft(b, 64, seed=args.seed)
    sd_dev = {k: getattr(sdraft, k).to(dev) for k in ("draft_tokens", "draft_logq", "topk_idx", "topk_q")}
    sp_outs = dipsd.spec_outputs(b.L, dev)
    ws_sp = dipsd.workspace(dipsd.dipsd_spec_verify_sparse_workspace_size(b.L, b.V), dev)

    def spec_sparse(k):
        c = copies[k % R]
        dipsd.dipsd_spec_verify_sparse(b.L, b.members, b.seed, c["z"], sd_dev["draft_tokens"], sd_dev["draft_logq"],
                                       sd_dev["topk_idx"], sd_dev["topk_q"], outputs=sp_outs, ws=ws_sp)

    def attn_append(k):
        c = copies[k % R]
        dipsd.dipsd_verify_attention_append(b.L, b.ctx, c["q"], new_k, new_v, c["kc"], c["vc"], bt, b.scale,
                                            out=attn_out, ws=ws)

    def cold_latency(fn, k):
        """Single calls with L2 flushed (a 256 MB write) before each, outside the events."""
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(k)]
        for i in range(k):
            flush.fill_(i & 0xFF)
            evs[i][0].record(stream)
            fn(i)
            evs[i][1].record(stream)
        torch.cuda.synchronize()
        return float(np.median([s_.elapsed_time(e_) for s_, e_ in evs]))

    for i in range(max(3, args.warmup)):
        step(i)
        attn_only(i)
        spec_only(i)
    torch.cuda.synchronize()
    assert dipsd.device_status(ws) == 0

    n_steps = args.steps
    g_step, launches = capture(step, n_steps, R, stream)

    sampler = ClockSampler(local)
    sampler.start()
    # the headline: replays of exactly K steps, as many on every rank (the
    # count agreed before timing), median over the replays
    first = replay_ms(g_step, stream, 2, barrier)[1]
    reps = max(3, min(2000, math.ceil(args.min_replay_ms / max(first, 1e-3))))
    if world > 1:
        t = torch.tensor([reps], device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        reps = int(t.item())
    step_ms = np.asarray(replay_ms(g_step, stream, reps, barrier))
    total_ms = float(np.median(step_ms))

    stages = {}
    for name, fn in (("verify_attention", attn_only), ("spec_verify", spec_only),
                     ("verify_attention_append", attn_append), ("spec_verify_sparse", spec_sparse)):
        g, _ = capture(fn, n_steps, R, stream)
        stages[name] = replay_stats(g, n_steps, stream, args.min_replay_ms / 3)
        del g
    lat_step = cold_latency(step, min(args.steps, 50))

    # end to end through the Python API: every step copies its inputs from
    # pinned host memory into one of R device slots (copy stream), makes the
    # call and reads its results back into that slot's pinned buffer (compute
    # stream); step k+1's upload overlaps step k's compute.  A slot's inputs
    # (q, target and draft logits, drafted tokens) sit back to back in one
    # device buffer, and the results (accept_len, out_offsets, out_tokens) in
    # another, so each step is one host-to-device and one device-to-host copy.
    h_in, views_of = packed_layout([b.q, b.target_logits, b.draft_logits, b.draft_tokens])
    h_in = h_in.pin_memory()
    d_in = [torch.empty_like(h_in, device=dev) for _ in range(R)]
    e_in = [dict(zip(("q", "z", "w", "d"), views_of(x))) for x in d_in]
    o_host, o_views = packed_layout([x.cpu() for x in outs[:3]])
    d_out = torch.empty_like(o_host, device=dev)
    e_outs = tuple(o_views(d_out)) + (outs[3],)
    h_out = [torch.empty_like(o_host).pin_memory() for _ in range(R)]
    h2d, d2h = h_in.numel(), d_out.numel()  # bytes copied per step (the packed buffers)
    cs = torch.cuda.Stream()
    ev_up = [torch.cuda.Event() for _ in range(R)]
    ev_free = [torch.cuda.Event() for _ in range(R)]
    api_s = [0.0]

    def e2e_steps(n, host_clock=False):
        cur = torch.cuda.current_stream()  # the compute stream (a capture's stream inside one)
        cs.wait_stream(cur)
        for i in range(n):
            k = i % R
            c = e_in[k]
            if i >= R:
                cs.wait_event(ev_free[k])
            with torch.cuda.stream(cs):
                d_in[k].copy_(h_in, non_blocking=True)
            ev_up[k].record(cs)
            cur.wait_event(ev_up[k])
            t0 = time.perf_counter()
            dipsd.dipsd_verify_batch(b.members, b.L, b.ctx, c["q"], copies[k]["kc"], copies[k]["vc"], bt, b.scale,
                                     c["z"], c["w"], c["d"], b.seed, attn_out=attn_out, outputs=e_outs, ws=ws,
                                     stream=cur)
            if host_clock:
                api_s[0] += time.perf_counter() - t0
            h_out[k].copy_(d_out, non_blocking=True)
            ev_free[k].record(cur)
        cur.wait_stream(cs)

    # plain calls: the library's host work (validation, planning, launches)
    # and the binding's argument marshalling are inside the timed region
    e2e_steps(R)
    torch.cuda.synchronize()
    if barrier:
        barrier()
    t0 = time.perf_counter()
    e2e_steps(n_steps, host_clock=True)
    torch.cuda.synchronize()
    e2e_plain_ms = 1000 * (time.perf_counter() - t0) / n_steps
    api_us = 1e6 * api_s[0] / n_steps
    # the same steps captured as one CUDA graph, replayed back to back (on a
    # stream that made plain calls first)
    g_e2e = torch.cuda.CUDAGraph()
    cap = torch.cuda.Stream()
    cap.wait_stream(stream)
    with torch.cuda.stream(cap):
        e2e_steps(R)
    torch.cuda.synchronize()
    with torch.cuda.graph(g_e2e, stream=cap):
        e2e_steps(R)
    g_e2e.replay()
    torch.cuda.synchronize()
    reps_g = max(1, n_steps // R)
    t0 = time.perf_counter()
    for _ in range(reps_g):
        g_e2e.replay()
    torch.cuda.synchronize()
    e2e_graph_ms = 1000 * (time.perf_counter() - t0) / (reps_g * R)
    clocks = sampler.stop()

    emitted = int(outs[1][-1].item())
    units = emitted * n_steps
    from paper_2604_20919_gb300.shard import aggregate_timing
    total_ms_max, units_all, e2e_max = aggregate_timing(total_ms, units, e2e_plain_ms * n_steps, device=dev)
    extra = {}
    if args.extra and world == 1:
        del g_step, g_e2e
        del copies, new_k, new_v, flush
        torch.cuda.empty_cache()
        for wl in (3, 4):
            if wl != args.workload:
                extra[f"stages_workload{wl}"] = measure_workload(wl, args, dev, stream, hbm_peak)
        extra["workload5"] = measure_pipeline(args, dev)
    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return
    write_line(args, b, world, hbm_peak, peak_kind, stages, total_ms_max, units_all, n_steps, step_ms, emitted,
               launches, lat_step, e2e_max, e2e_graph_ms, api_us, h2d, d2h, clocks, extra, R)
    if world > 1:
        dist.destroy_process_group()


def write_line(args, b, world, hbm_peak, peak_kind, stages, total_ms_max, units_all, n_steps, step_ms, emitted,
               launches, lat_step, e2e_max, e2e_graph_ms, api_us, h2d, d2h, clocks, extra, R):
    a_bytes, s_bytes = attention_bytes(b), spec_bytes(b)
    stages["verify_attention"] = stage_entry(stages["verify_attention"], a_bytes, hbm_peak)
    stages["spec_verify"] = stage_entry(stages["spec_verify"], s_bytes, hbm_peak)
    stages["spec_verify_sparse"] = dict(stage_entry(stages["spec_verify_sparse"], sparse_bytes(b), hbm_peak),
                                        note="sparse draft payload, K = 64 table entries per draft row")
    stages["verify_attention_append"]["note"] = ("attention that also writes the verify tokens' K/V rows into "
                                                 "their pages (same launch)")
    # The roofline is the single kernel with the longest launches: the attention
    # kernel (one launch per stage on this workload), ahead of each of the
    # three chained spec-verify kernels (see the ncu launch list under profiles/).
    dom = "verify_attention"
    ds = stages[dom]
    traffic = recorded_traffic(dom, args.workload, source_hash(["paper_2604_20919_gb300/csrc/attention_tc.cuh"]))
    ms_attn, ms_spec = stages["verify_attention"]["ms"], stages["spec_verify"]["ms"]
    per_step = step_ms / n_steps
    line = {
        "metric": "verified tokens/s (one verification stage: attention + speculative sampling)",
        "value": units_all / (total_ms_max / 1000.0),
        "unit": "verified tokens/s",
        "n_gpus": world, "steps": n_steps, "warmup": args.warmup,
        "ms_per_step": total_ms_max / n_steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic",
        "config": bench_config(b, args.workload, args.seed, world),
        "timing": {"replays": int(len(step_ms)), "steps_per_replay": n_steps,
                   "ms_per_step_median": float(np.median(per_step)), "ms_per_step_min": float(per_step.min()),
                   "ms_per_step_max": float(per_step.max()),
                   "note": "value = median replay; every replay times exactly `steps` steps between CUDA events"},
        "emitted_tokens_per_step": emitted,
        "roofline": {"kernel": dom, "bound": "hbm", "achieved": ds["gbs"], "peak": hbm_peak, "unit": "GB/s",
                     "frac": ds["gbs"] / hbm_peak, "peak_kind": peak_kind, "traffic": traffic,
                     "alg_bytes_per_launch": ds["alg_bytes"]},
        "stages": stages,
        "projection_64_layer_attention": {
            "value": emitted / ((64 * ms_attn + ms_spec) / 1000.0), "unit": "verified tokens/s",
            "note": "64 attention layers (each timed like verify_attention) + spec_verify; excludes every GEMM"},
        "step_latency_cold_l2_ms": lat_step,
        "e2e": {"value": units_all / (e2e_max / 1000.0),
                "unit": "verified tokens/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "ms_per_step": e2e_max / n_steps, "api_host_us_per_call": api_us,
                "schedule": "plain calls through the Python API (the library's validation and planning included); "
                            "per step: one pinned H2D copy of q, logits and drafts (packed) on a copy stream; "
                            "the call; one D2H copy of accept_len, offsets, tokens (packed); uploads overlap "
                            "the previous step's compute; host clock"},
        "e2e_graph": {"value": emitted / (e2e_graph_ms / 1000.0), "unit": "verified tokens/s",
                      "ms_per_step": e2e_graph_ms,
                      "schedule": "the same steps captured as one CUDA graph of the API calls, replayed back to back"},
        "gpu_launches": int(launches),
        "clocks": clocks,
    }
    line.update(extra)
    if world == 1 and args.cpu_seconds > 0:
        line["cpu_baseline"] = cpu_baseline(b, args.cpu_seconds)
    print(json.dumps(line), flush=True)


def measure_pipeline(args, dev):
    """Workload 5: 128 users in one KV pool dealt into 4 stages of 32, each stage
    one dipsd_verify_batch, stages alternating over two streams and rounds
    repeating back to back (one CUDA graph); the sustained verified tokens/s."""
    import torch
    from paper_2604_20919_gb300 import dipsd
    from workloads import make_config, config_shape, CONFIG_NAMES

    batches = make_config(5, seed=args.seed, device="cpu", kv_device=dev)
    s = config_shape(5, args.seed)
    L_all, ctx_all = s["L"], s["ctx"]
    kc, vc = batches[0].k_cache, batches[0].v_cache
    bt = batches[0].block_table.to(dev)
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    stage = []
    for n, b in enumerate(batches):
        g = lambda t: t.to(dev)
        ws = dipsd.workspace(dipsd.dipsd_verify_batch_workspace_size(b.members, L_all, ctx_all, b.Hq, b.Hkv, b.D,
                                                                     b.V), dev)
        stage.append(dict(b=b, q=g(b.q), z=g(b.target_logits), w=g(b.draft_logits), d=g(b.draft_tokens),
                          attn=torch.empty_like(b.q, device=dev),
                          outs=dipsd.spec_outputs(b.L, dev), ws=ws, stream=streams[n % 2]))
    main = torch.cuda.current_stream()

    def rounds(k):
        cur = torch.cuda.current_stream()  # the capture stream inside a graph capture
        for sm in streams:
            sm.wait_stream(cur)
        for _ in range(k):
            for x in stage:
                with torch.cuda.stream(x["stream"]):
                    dipsd.dipsd_verify_batch(x["b"].members, L_all, ctx_all, x["q"], kc, vc, bt, x["b"].scale,
                                             x["z"], x["w"], x["d"], x["b"].seed, attn_out=x["attn"],
                                             outputs=x["outs"], ws=x["ws"], stream=x["stream"])
        for sm in streams:
            cur.wait_stream(sm)

    k = 20
    rounds(1)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    n0 = dipsd.dipsd_launch_count()
    with torch.cuda.graph(graph):
        rounds(k)
    launches = dipsd.dipsd_launch_count() - n0
    graph.replay()
    torch.cuda.synchronize()
    first = replay_ms(graph, main, 1)[0]
    reps = max(3, min(500, math.ceil(args.min_replay_ms / max(first, 1e-3))))
    t = np.asarray(replay_ms(graph, main, reps)) / k
    ms = float(np.median(t))
    emitted = sum(int(x["outs"][1][-1].item()) for x in stage)
    kv_bytes = sum(attention_bytes(x["b"]) for x in stage)
    assert all(dipsd.device_status(x["ws"]) == 0 for x in stage)
    res = {
        "metric": "verified tokens/s (sustained: 4 pipeline stages of 32 users on two streams)",
        "value": emitted / (ms / 1000.0), "unit": "verified tokens/s", "ms_per_round": ms,
        "ms_per_round_min": float(t.min()), "ms_per_round_max": float(t.max()), "replays": reps,
        "rounds_per_replay": k, "config": {"workload": CONFIG_NAMES[5], "stages": 4, "users_per_stage": 32,
                                           "streams": 2, "l2": "2 GB KV pool read once per round (>> L2)"},
        "attention_gbs": kv_bytes / (ms / 1000.0) / 1e9,
        "emitted_tokens_per_round": emitted, "gpu_launches_per_replay": launches,
    }
    del stage, kc, vc, batches
    torch.cuda.empty_cache()
    return res


def run_pipeline(args):
    """`--workload 5`: the pipelined schedule's sustained rate as its own line."""
    import torch
    from paper_2604_20919_gb300 import dipsd
    if int(os.environ.get("RANK", "0")) != 0:
        return
    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", "0")))
    torch.cuda.set_device(dev)
    dipsd.load()
    res = measure_pipeline(args, dev)
    res.update({"n_gpus": 1, "steps": res["rounds_per_replay"], "warmup": args.warmup, "higher_is_better": True,
                "dtype": "bf16", "data": "synthetic"})
    print(json.dumps(res), flush=True)


def main():
    args = parse_args()
    if args.impl == "reference":
        run_reference(args)
    elif args.workload == 5:
        run_pipeline(args)
    else:
        run_dipsd(args)


if __name__ == "__main__":
    main()
