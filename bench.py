#!/usr/bin/env python
"""Verified tokens/s of DiP-SD batch verification on one GB300 (and per-stage HBM roofline).

One step = one pipeline stage verified end to end on the GPU through the C ABI
(dipsd_verify_batch: verify attention over every user's paged KV cache, then
speculative sampling over the vocabulary) on the Qwen3-32B-shaped batch
(B=8, L_i ~ U{1..8}, context 1024, 64/8/128 heads, V=151936).  Inputs are
resident in HBM; L2 is flushed (a 256 MB write) between timed steps, outside
the timed events.  The line also carries the end-to-end number through the
same call with host buffers (copies inside the timed region), per-stage
roofline figures against the measured HBM copy bandwidth, the clocks seen
while timing, and the fp64 CPU oracle timed on the host cores.

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
FALLBACK_HBM_GBS = 6800.0


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["dipsd", "reference"], default="dipsd")
    ap.add_argument("--workload", type=int, default=2, help="workload id (2 = the headline batch)")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--cpu-seconds", type=float, default=10.0, help="budget of the CPU oracle baseline")
    return ap.parse_args()


def workload_config(b, wl, seed):
    from workloads import CONFIG_NAMES
    return {"workload": CONFIG_NAMES[wl], "B": int(b.B), "L": [int(x) for x in b.L],
            "ctx": [int(x) for x in b.ctx], "heads": f"{b.Hq}/{b.Hkv}/{b.D}", "V": int(b.V),
            "page": 16, "seed": seed, "l2": "flushed between timed steps (256 MB write)"}


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


def source_hash(paths):
    h = hashlib.sha256()
    for p in paths:
        with open(os.path.join(ROOT, p), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel_file, src_hash):
    """DRAM bytes per launch from the committed ncu summary, if taken on this source."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f).get(kernel_file)
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
    if rank != 0:
        return
    import torch
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
            "config": workload_config(b, args.workload, args.seed), "impl": "reference",
            "cpu_baseline": {"value": value, "unit": "verified tokens/s", "cores": os.cpu_count(),
                             "kind": "oracle", "sample": f"{args.steps} full batch(es) of the workload"},
            "e2e": {"value": value, "unit": "verified tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


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
    dipsd.load()

    # each rank verifies its own replica (independent users): weak scaling, no collective
    b = make_config(args.workload, seed=args.seed + rank, device="cpu", kv_device=dev)
    q, z, w = b.q.to(dev), b.target_logits.to(dev), b.draft_logits.to(dev)
    d, u, bt = b.draft_tokens.to(dev), b.uniforms.to(dev), b.block_table.to(dev)
    kc, vc = b.k_cache, b.v_cache
    attn_out = torch.empty_like(q)
    outs = dipsd.spec_outputs(b.L, dev)
    ws = dipsd.workspace(dipsd.dipsd_verify_batch_workspace_size(b.members, b.L, b.ctx, b.Hq, b.Hkv, b.D, b.V), dev)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    def step():
        dipsd.dipsd_verify_batch(b.members, b.L, b.ctx, q, kc, vc, bt, b.scale, z, w, d, u, attn_out=attn_out,
                                 outputs=outs, ws=ws)

    def attn_only():
        dipsd.dipsd_verify_attention(b.L, b.ctx, q, kc, vc, bt, b.scale, out=attn_out, ws=ws)

    def spec_only():
        dipsd.dipsd_spec_verify(b.L, z, w, d, u, outputs=outs, ws=ws)

    def timed(fn, k):
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(k)]
        for i in range(k):
            flush.fill_(i & 0xFF)
            evs[i][0].record(stream)
            fn()
            evs[i][1].record(stream)
        torch.cuda.synchronize()
        return np.array([s.elapsed_time(e) for s, e in evs])

    for _ in range(max(3, args.warmup)):
        step()
        attn_only()
        spec_only()
    torch.cuda.synchronize()
    assert dipsd.device_status(ws) == 0

    sampler = ClockSampler(local)
    sampler.start()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    n0 = dipsd.dipsd_launch_count()
    t_step = timed(step, args.steps)
    launches = dipsd.dipsd_launch_count() - n0
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    t_attn = timed(attn_only, args.steps)
    t_spec = timed(spec_only, args.steps)

    # end to end through the same call: pinned host inputs in, emitted tokens out
    pin = lambda t: t.cpu().pin_memory()
    h_in = [pin(x) for x in (b.q, b.target_logits, b.draft_logits, b.draft_tokens, b.uniforms)]
    d_in = [q, z, w, d, u]
    h_out = [torch.empty_like(x, device="cpu").pin_memory() for x in outs[:3]]
    h2d = sum(x.numel() * x.element_size() for x in h_in)
    d2h = sum(x.numel() * x.element_size() for x in h_out)
    e2e_ms = []
    for i in range(args.steps):
        flush.fill_(i & 0xFF)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for hd, dd in zip(h_in, d_in):
            dd.copy_(hd, non_blocking=True)
        step()
        for hd, dd in zip(h_out, outs[:3]):
            hd.copy_(dd, non_blocking=True)
        stream.synchronize()
        e2e_ms.append(1000 * (time.perf_counter() - t0))
    clocks = sampler.stop()

    emitted = int(outs[1][-1].item())
    total_ms = float(t_step.sum())
    units = emitted * args.steps
    if world > 1:
        tt = torch.tensor([total_ms, units, float(np.sum(e2e_ms))], dtype=torch.float64, device=dev)
        mx = tt.clone()
        dist.all_reduce(mx, op=dist.ReduceOp.MAX)
        dist.all_reduce(tt, op=dist.ReduceOp.SUM)
        total_ms_max, units_all, e2e_max = float(mx[0]), float(tt[1]), float(mx[2])
    else:
        total_ms_max, units_all, e2e_max = total_ms, float(units), float(np.sum(e2e_ms))
    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return

    hbm_peak, peak_kind = read_peaks()
    a_bytes, s_bytes = attention_bytes(b), spec_bytes(b)
    a_ms, s_ms = float(t_attn.mean()), float(t_spec.mean())
    stages = {
        "verify_attention": {"ms": a_ms, "alg_bytes": a_bytes, "gbs": a_bytes / a_ms / 1e6,
                             "frac_of_measured_hbm": a_bytes / a_ms / 1e6 / hbm_peak,
                             "frac_of_8000": a_bytes / a_ms / 1e6 / 8000.0},
        "spec_verify": {"ms": s_ms, "alg_bytes": s_bytes, "gbs": s_bytes / s_ms / 1e6,
                        "frac_of_measured_hbm": s_bytes / s_ms / 1e6 / hbm_peak,
                        "frac_of_8000": s_bytes / s_ms / 1e6 / 8000.0},
    }
    dom = "verify_attention" if a_ms >= s_ms else "spec_verify"
    src = {"verify_attention": ["paper_2604_20919_gb300/csrc/attention.cuh"],
           "spec_verify": ["paper_2604_20919_gb300/csrc/spec_verify.cuh"]}[dom]
    ds = stages[dom]
    traffic = recorded_traffic(dom, source_hash(src))
    line = {
        "metric": "verified tokens/s (one verification stage: attention + speculative sampling)",
        "value": units_all / (total_ms_max / 1000.0),
        "unit": "verified tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": total_ms_max / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic",
        "config": dict(workload_config(b, args.workload, args.seed),
                       parallelism="replicas" if world > 1 else "single"),
        "emitted_tokens_per_step": emitted,
        "roofline": {"kernel": dom, "bound": "hbm", "achieved": ds["gbs"], "peak": hbm_peak, "unit": "GB/s",
                     "frac": ds["gbs"] / hbm_peak, "peak_kind": peak_kind, "traffic": traffic,
                     "alg_bytes_per_launch": ds["alg_bytes"]},
        "stages": stages,
        "e2e": {"value": units_all / (e2e_max / 1000.0), "unit": "verified tokens/s",
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "ms_per_step": e2e_max / args.steps},
        "gpu_launches": int(launches),
        "clocks": clocks,
        "step_ms_p50": float(np.median(t_step)), "step_ms_min": float(t_step.min()),
    }
    if world == 1:
        line["cpu_baseline"] = cpu_baseline(b, args.cpu_seconds)
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def main():
    args = parse_args()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_dipsd(args)


if __name__ == "__main__":
    main()
