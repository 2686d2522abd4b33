"""Benchmark of the end-of-prefill diversified KV-eviction step on GB300.

One step = the whole path for one request of the Mistral-7B-shaped workload
"mistral-32layer-L32768-B64": 32 layers x 8 KV heads (256 units), prefix 32768,
window 32, budget 64, lambda = (0.5, -0.5): score (window attention, mu, sigma),
select (pooling, top-4B, greedy MMR) and gather (compact K/V cache).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

N > 1 runs under torchrun, one rank per GPU; every rank evicts its own request
(weak scaling, no collective on the data path). Rank 0 prints one JSON line.
--impl reference times the fp64 CPU oracle (the only reference this path has) on
a bounded sample of the same workload on the host cores.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = "mistral-32layer-L32768-B64"
METRIC = "eviction-step ms/request (32 layers) & prefix tok/s; % of HBM roofline"
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_HBM_GBS = 6800.0

# DRAM traffic of one score-kernel launch (dram__bytes_read.sum + dram__bytes_write.sum),
# from the ncu capture summarised in profiles/, valid only for the sources it was taken
# on (sha256 over csrc/kve_score.cu and csrc/kve_host.cu, which sets the schedule); per
# launch of the full workload.
SCORE_TRAFFIC = {"source_sha256": "6593b248e96b4d98f638c81c75750ae26af939cef30a1c7eb39fbcb49690d658",
                 "bytes_per_launch": 2178506496 + 75100672}


def _score_source_sha():
    h = hashlib.sha256()
    for f in ("kve_score.cu", "kve_host.cu"):
        h.update(open(os.path.join(ROOT, "paper_2609_30738_gb300", "csrc", f), "rb").read())
    return h.hexdigest()


def _peaks():
    try:
        d = json.load(open(PEAKS_FILE))
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def _dist():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def _max_over_ranks(x, world, device):
    """Job time = the slowest rank's time (every rank holds the max afterwards)."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def _job_tok_s(world, prefix_len, step_s):
    """Whole-job throughput: every rank evicts one request of prefix_len tokens per step."""
    return world * prefix_len / step_s


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.t0 = self.t1 = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "50", "-i", str(self.gpu)], stdout=subprocess.PIPE,
                stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        time.sleep(0.3)

    def mark(self, which):
        setattr(self, which, time.time())

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        out, _ = self.proc.communicate(timeout=10)
        rows = [r.split(", ") for r in out.strip().splitlines() if r.strip()]
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            try:
                sm.append(float(r[1]))
                mx = float(r[2])
                for nm, val in zip(names, r[5:9]):
                    if val.strip().lower() == "active":
                        reasons.add(nm)
            except (ValueError, IndexError):
                continue
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------------ oracle baseline


_SAMPLE = None


def _oracle_init(path, n_units, q_shape, k_shape, meta):
    """Worker initialiser: map the shared sample file (no copies per task)."""
    global _SAMPLE
    qn = int(np.prod(q_shape))
    kn = int(np.prod(k_shape))
    mm = np.memmap(path, dtype=np.uint16, mode="r", shape=(n_units, qn + kn))
    _SAMPLE = (mm, q_shape, k_shape, meta)


def _oracle_unit(u):
    """Score and select one unit with the fp64 oracle (runs in a spawned worker)."""
    from oracle import kv_evict_oracle as O
    mm, q_shape, k_shape, (L, W, G, B, l1, l2) = _SAMPLE
    qn = int(np.prod(q_shape))
    q_bits = np.asarray(mm[u, :qn]).reshape(q_shape)
    k_bits = np.asarray(mm[u, qn:]).reshape(k_shape)
    t = time.perf_counter()
    O.evict_unit(q_bits, k_bits, L, W, G, B, l1, l2)
    return time.perf_counter() - t


class OraclePool:
    """Spawned worker processes (one BLAS thread each) over a memory-mapped sample."""

    def __init__(self, spec, sample, workers):
        import multiprocessing as mp
        import tempfile
        for var in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
            os.environ[var] = "1"
        G = spec["num_q_heads"] // spec["num_kv_heads"]
        q_shape, k_shape = sample[0][0].shape, sample[0][1].shape
        self.dir = tempfile.mkdtemp(prefix="kve_oracle_")
        self.path = os.path.join(self.dir, "sample.u16")
        n = len(sample)
        mm = np.memmap(self.path, dtype=np.uint16, mode="w+",
                       shape=(n, int(np.prod(q_shape)) + int(np.prod(k_shape))))
        for i, (q, k) in enumerate(sample):
            mm[i] = np.concatenate([q.reshape(-1), k.reshape(-1)])
        mm.flush()
        del mm
        meta = (spec["seq_lens"][0], spec["window"], G, spec["budget"], 0.5, -0.5)
        self.n = n
        self.pool = mp.get_context("spawn").Pool(
            workers, initializer=_oracle_init, initargs=(self.path, n, q_shape, k_shape, meta))

    def run(self):
        """Wall time of one pass over every unit of the sample."""
        t = time.perf_counter()
        self.pool.map(_oracle_unit, range(self.n), chunksize=1)
        return time.perf_counter() - t

    def close(self):
        self.pool.close()
        self.pool.join()
        try:
            os.remove(self.path)
            os.rmdir(self.dir)
        except OSError:
            pass


def _oracle_sample_from_host(spec, n_units, seed):
    """(q_bits, k_bits) of the first n_units units, generated on the CPU."""
    import torch
    from paper_2609_30738_gb300 import synth
    from tests.parity import to_bits
    G = spec["num_q_heads"] // spec["num_kv_heads"]
    W, L, Hkv = spec["window"], spec["seq_lens"][0], spec["num_kv_heads"]
    out = []
    layer = 0
    while len(out) < n_units:
        k, v, q = synth.unit_tensors(seed, 0, layer, L, Hkv, G, W,
                                     salient_frac=spec.get("salient_frac", 0.0))
        for h in range(Hkv):
            if len(out) < n_units:
                out.append((to_bits(q[h].to(torch.bfloat16)), to_bits(k[h].to(torch.bfloat16))))
        layer += 1
    return out


def run_reference(args):
    """--impl reference: the fp64 oracle on the host cores, bounded sample per step."""
    world, rank, _ = _dist()
    if rank != 0:
        return
    from paper_2609_30738_gb300.workloads import WORKLOADS
    spec = WORKLOADS[WORKLOAD]
    cores = os.cpu_count() or 1
    n_units = cores          # one unit per host core and step
    sample = _oracle_sample_from_host(spec, n_units, 2609)
    pool = OraclePool(spec, sample, cores)
    try:
        for _ in range(args.warmup):
            pool.run()
        times = [pool.run() for _ in range(args.steps)]
    finally:
        pool.close()
    step_s = sum(times) / len(times)
    units_total = spec["num_layers"] * spec["num_kv_heads"]
    L = spec["seq_lens"][0]
    tok_s = L * (n_units / units_total) / step_s
    ms_req = step_s * 1e3 * units_total / n_units
    line = {"impl": "reference", "metric": METRIC, "value": tok_s, "unit": "prefix tok/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": ms_req, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOAD, "sample_units": n_units},
            "cpu_baseline": {"value": tok_s, "unit": "prefix tok/s", "cores": cores, "kind": "oracle",
                             "sample": f"{n_units} of 256 units (score + select) per step, "
                                       "extrapolated to the 256-unit request"},
            "e2e": {"value": tok_s, "unit": "prefix tok/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------ GPU arm


def run_ours(args):
    import torch
    import torch.distributed as dist
    from paper_2609_30738_gb300 import kv_evict as K
    from paper_2609_30738_gb300 import synth
    from paper_2609_30738_gb300.workloads import WORKLOADS, lambda_arrays

    world, rank, local = _dist()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    spec = WORKLOADS[WORKLOAD]
    if args.layers:
        spec = dict(spec, num_layers=args.layers)
    L = spec["seq_lens"][0]
    W, B, d = spec["window"], spec["budget"], spec["head_dim"]
    N_L, Hkv = spec["num_layers"], spec["num_kv_heads"]
    units = N_L * Hkv

    # inputs resident in HBM: each rank evicts its own request (seeded by rank)
    batch = synth.make_batch(spec, seed=2609 + rank, device=dev)
    q, k, v = batch["q_win"], batch["k"], batch["v"]
    plan = K.Plan(spec, batch["seq_lens"])
    bufs = K.Buffers(plan, device=dev, with_trace=False)
    lam1, lam2 = lambda_arrays(spec, K.profile)
    stream = torch.cuda.Stream(device=dev)

    def step():
        K.run_step(plan, bufs, q, k, v, lam1, lam2, stream=stream)

    # correctness of the timed configuration: device status after a first step
    with torch.cuda.stream(stream):
        step()
    if plan.status(bufs.ws, stream) != K.KVE_OK:
        raise RuntimeError("device-side wait timed out")

    for _ in range(args.warmup):
        step()
    stream.synchronize()

    sampler = ClockSampler(local) if rank == 0 else None
    if sampler:
        sampler.start()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    if sampler:
        sampler.mark("t0")
    t0.record(stream)
    for i in range(args.steps):
        ev[i][0].record(stream)
        plan.score(q, k, bufs.mu, bufs.sigma, bufs.ws, stream)
        ev[i][1].record(stream)
        plan.select(bufs.mu, bufs.sigma, k, lam1, lam2, bufs.indices, bufs.ws, None, None, stream)
        plan.gather(k, v, bufs.indices, bufs.k_out, bufs.v_out, stream)
    t1.record(stream)
    torch.cuda.synchronize()
    if sampler:
        sampler.mark("t1")
    if world > 1:
        dist.barrier()
    elapsed = t0.elapsed_time(t1) / 1e3
    score_s = sum(a.elapsed_time(b) for a, b in ev) / 1e3 / args.steps
    clocks = sampler.stop() if sampler else None
    if plan.status(bufs.ws, stream) != K.KVE_OK:
        raise RuntimeError("device-side wait timed out in the timed region")
    elapsed = _max_over_ranks(elapsed, world, dev)

    # end to end through the public API with host buffers (pinned), copies inside.
    # The request is evicted in chunks of layers, one plan per chunk: the copy stream
    # brings in chunk c + 1 while the compute stream scores, selects and gathers chunk
    # c (every array is layer-major for one request, so a chunk is a contiguous view).
    # V stays in pinned host memory: the gather reads the kept rows in place, so
    # min(B_l, L_r - W) + W rows per unit cross the host link, not the whole tensor.
    e2e = None
    if args.e2e_steps > 0:
        # layer chunks are contiguous views only for one request per plan
        chunks = (args.e2e_chunks if args.e2e_chunks > 0 and N_L % args.e2e_chunks == 0
                  and len(batch["seq_lens"]) == 1 else 1)
        Lc = N_L // chunks
        hq = q.cpu().pin_memory()
        hk = k.cpu().pin_memory()
        hv = v.cpu().pin_memory()
        o_idx = torch.empty_like(bufs.indices, device="cpu").pin_memory()
        o_k = torch.empty_like(bufs.k_out, device="cpu").pin_memory()
        o_v = torch.empty_like(bufs.v_out, device="cpu").pin_memory()
        dq, dk = torch.empty_like(q), torch.empty_like(k)
        cplan = K.Plan(dict(spec, num_layers=Lc), batch["seq_lens"])
        cws = torch.empty(cplan.workspace_bytes, dtype=torch.uint8, device=dev)
        mu_c = bufs.mu.view(chunks, -1)
        sg_c = bufs.sigma.view(chunks, -1)
        idx_c = bufs.indices.view(chunks, Lc * Hkv, -1)
        ko_c = bufs.k_out.view(chunks, Lc * Hkv, *bufs.k_out.shape[1:])
        vo_c = bufs.v_out.view(chunks, Lc * Hkv, *bufs.v_out.shape[1:])
        copy_stream = torch.cuda.Stream(device=dev)
        arrived = [torch.cuda.Event() for _ in range(chunks)]
        v_rows = sum(Hkv * (min(plan.layer_budgets[l], Lr - W) + W)
                     for Lr in plan.seq_lens for l in range(N_L))
        v_read = v_rows * d * hv.element_size()

        def e2e_step():
            copy_stream.wait_stream(stream)    # the previous step has finished with dq, dk
            with torch.cuda.stream(copy_stream):
                for c in range(chunks):
                    dq[c * Lc:(c + 1) * Lc].copy_(hq[c * Lc:(c + 1) * Lc], non_blocking=True)
                    dk[c * Lc:(c + 1) * Lc].copy_(hk[c * Lc:(c + 1) * Lc], non_blocking=True)
                    arrived[c].record(copy_stream)
            for c in range(chunks):
                ls = slice(c * Lc, (c + 1) * Lc)
                stream.wait_event(arrived[c])
                cplan.score(dq[ls], dk[ls], mu_c[c], sg_c[c], cws, stream)
                cplan.select(mu_c[c], sg_c[c], dk[ls], lam1[ls], lam2[ls], idx_c[c], cws, None, None,
                             stream)
                cplan.gather(dk[ls], hv[ls], idx_c[c], ko_c[c], vo_c[c], stream)
            with torch.cuda.stream(stream):
                o_idx.copy_(bufs.indices, non_blocking=True)
                o_k.copy_(bufs.k_out, non_blocking=True)
                o_v.copy_(bufs.v_out, non_blocking=True)

        for _ in range(2):                     # first touches of the pinned buffers
            e2e_step()
        stream.synchronize()
        if cplan.status(cws, stream) != K.KVE_OK:
            raise RuntimeError("device-side wait timed out in the end-to-end step")
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        if world > 1:
            dist.barrier()
        copy_stream.wait_stream(stream)
        a.record(copy_stream)
        for _ in range(args.e2e_steps):
            e2e_step()
        b.record(stream)
        torch.cuda.synchronize()
        if cplan.status(cws, stream) != K.KVE_OK:
            raise RuntimeError("device-side wait timed out in the end-to-end step")
        e2e_s = a.elapsed_time(b) / 1e3 / args.e2e_steps
        e2e_s = _max_over_ranks(e2e_s, world, dev)
        h2d = sum(x.numel() * x.element_size() for x in (hq, hk)) + v_read
        d2h = sum(x.numel() * x.element_size() for x in (o_idx, o_k, o_v))
        e2e = {"value": _job_tok_s(world, L, e2e_s), "unit": "prefix tok/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": e2e_s * 1e3, "layer_chunks": chunks,
               "v": "read in place from pinned host memory by the gather (kept rows only)"}
        del hq, hk, hv, dq, dk

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return

    # roofline of the dominant kernel (score): algorithmic bytes per launch
    n_rows = spec["num_q_heads"] // Hkv * W
    score_bytes = units * (L * d * 2 + n_rows * d * 2 + 2 * 4 * L)
    gather_bytes = units * 2 * 2 * (B + W) * d * 2
    peak, peak_kind = _peaks()
    achieved = score_bytes / score_s / 1e9
    traffic = (SCORE_TRAFFIC["bytes_per_launch"]
               if SCORE_TRAFFIC["source_sha256"] == _score_source_sha() else None)

    cpu = None
    if world == 1 and args.cpu_units > 0:
        cpu = cpu_baseline_from_device(spec, batch, args.cpu_units)

    step_s = elapsed / args.steps
    line = {"metric": METRIC, "value": _job_tok_s(world, L, step_s), "unit": "prefix tok/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": step_s * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16xbf16->f32", "data": "synthetic (seeded Mistral-7B-shaped K/V/Q)",
            "config": {"workload": WORKLOAD if not args.layers else f"{WORKLOAD} ({N_L} layers)",
                       "layers": N_L, "kv_heads": Hkv,
                       "q_heads": spec["num_q_heads"], "head_dim": d, "prefix_len": L,
                       "window": W, "budget": B, "lambda1": 0.5, "lambda2": -0.5,
                       "pool_kernel": spec["pool_kernel"], "requests_per_gpu": 1,
                       "l2": "inputs larger than L2 (2.15 GB of K read per step)"},
            "ms_per_request": step_s * 1e3,
            "hbm_roofline_frac_step": (score_bytes + gather_bytes) / step_s / 1e9 / peak,
            "score_kernel_ms": score_s * 1e3,
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak, "traffic": traffic,
                         "peak_source": peak_kind, "kernel": "kve score_kernel",
                         "algorithmic_bytes_per_launch": score_bytes},
            "gpu_launches": 3 * args.steps,
            "clocks": clocks, "cpu_baseline": cpu, "e2e": e2e}
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def cpu_baseline_from_device(spec, batch, n_units):
    """Oracle on the first n_units units of the device-resident inputs."""
    from tests.parity import to_bits
    G = spec["num_q_heads"] // spec["num_kv_heads"]
    W, Hkv = spec["window"], spec["num_kv_heads"]
    sample = []
    for u in range(n_units):
        layer, h = divmod(u, Hkv)
        sample.append((to_bits(batch["q_win"][layer, 0, h * G:(h + 1) * G]).reshape(G * W, -1),
                       to_bits(batch["k"][layer, h])))
    cores = min(os.cpu_count() or 1, n_units)
    pool = OraclePool(spec, sample, cores)
    try:
        wall = pool.run()
    finally:
        pool.close()
    units_total = spec["num_layers"] * Hkv
    L = spec["seq_lens"][0]
    return {"value": L * (n_units / units_total) / wall, "unit": "prefix tok/s", "cores": cores,
            "kind": "oracle",
            "sample": f"{n_units} of {units_total} units (score + select), wall {wall:.1f} s on "
                      f"{cores} worker processes, extrapolated to the whole request"}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=500)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--e2e-steps", type=int, default=5)
    ap.add_argument("--e2e-chunks", type=int, default=8,
                    help="layer chunks of the end-to-end step (copy of chunk c+1 beside compute of c)")
    ap.add_argument("--cpu-units", type=int, default=128)
    ap.add_argument("--layers", type=int, default=0,
                    help="profiling only: fewer layers than the workload (0 = all)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
