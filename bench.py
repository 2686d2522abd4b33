"""Benchmark of the end-of-prefill diversified KV-eviction step on GB300.

One step = the whole path for one call of a Mistral-7B-shaped workload: score
(window attention, mu, sigma), then select (pooling, top-4B, greedy MMR) with the
gather (compact K/V cache) in the same launch. Beside the step the line reports the
window-output pass, the one-pass score given the window rows' normalisers, the end-to-
end call from host buffers and the oracle's throughput. The default workload is
"mistral-32layer-L32768-B64": one
request of 32 layers x 8 KV heads (256 units), prefix 32768, window 32, budget 64,
lambda = (0.5, -0.5). --workload names any of the full-size workloads.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--workload NAME]

N > 1 runs under torchrun, one rank per GPU, with no collective on the data path.
A one-request workload gives every rank its own request (weak scaling); the
16-request batch is split across the ranks by prefix tokens (strong scaling).
Rank 0 prints one JSON line. --impl reference times the fp64 CPU oracle (the only
reference this path has) on a bounded sample of the same workload on the host
cores.
"""

from __future__ import annotations

import argparse
import gc
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
BENCH_WORKLOADS = ("mistral-32layer-L8192", "mistral-32layer-L32768-B32", "mistral-32layer-L32768-B64",
                   "mistral-32layer-L32768-B128", "mistral-32layer-L16384-segments",
                   "mistral-32layer-ragged16")
METRIC = "eviction-step ms/request (32 layers) & prefix tok/s; % of HBM roofline"
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_HBM_GBS = 6800.0

# DRAM traffic of one score-kernel launch (dram__bytes_read.sum + dram__bytes_write.sum),
# from the ncu capture summarised in profiles/, valid only for the sources it was taken
# on (sha256 over csrc/kve_score.cu and csrc/kve_host.cu, which sets the schedule); per
# launch of the full workload.
SCORE_TRAFFIC = {"source_sha256": "60b3a57416c0a61c7b7c3b1774a219755c992425eaef2ae96c39b9cac38a0974",
                 "bytes_per_launch": 2172808960 + 74820352}


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


def _rank_requests(spec, world, rank):
    """(request ids this rank evicts, scaling). A one-request workload: every rank
    its own request (id = rank), weak scaling. A batch: the batch's requests split
    across the ranks by prefix tokens, strong scaling."""
    from paper_2609_30738_gb300.workloads import partition_requests
    if len(spec["seq_lens"]) == 1:
        return [rank], "weak"
    return partition_requests(spec["seq_lens"], world)[rank], "strong"


def _config(name, spec, world):
    """The `config` object of both arms' JSON lines (identical for the same workload
    and number of GPUs)."""
    seq = spec["seq_lens"]
    scaling = "weak" if len(seq) == 1 else "strong"
    return {"workload": name, "parallelism": f"{scaling} x{world} (requests per rank, no collective)",
            "requests_per_step_job": world if scaling == "weak" else len(seq), "layers": spec["num_layers"], "kv_heads": spec["num_kv_heads"],
            "q_heads": spec["num_q_heads"], "head_dim": spec["head_dim"],
            "prefix_len": seq[0] if len(seq) == 1 else f"{len(seq)} requests, {min(seq)}-{max(seq)}",
            "tokens_per_call": sum(seq), "window": spec["window"], "budget": spec["budget"],
            "lambdas": list(spec["lambdas"][:1]) + [str(x) for x in spec["lambdas"][1:]],
            "pool_kernel": spec["pool_kernel"],
            "l2": "inputs larger than L2 (the K read per step exceeds 129 MB)"}


def _algorithmic_bytes(spec, seq, layer_budgets):
    """Algorithmic bytes of one step (bytes that must cross HBM): K read once
    (L d 2 per unit) by the score kernel; K and V rows gathered (min(B_l, L - W) + W
    rows read per unit and B + W rows written, K and V). Secondary traffic, not
    counted: the window queries (n d 2 per unit) and the mu / sigma writes (8 L)."""
    N_L, Hkv, W, B, d = (spec["num_layers"], spec["num_kv_heads"], spec["window"], spec["budget"],
                         spec["head_dim"])
    n = spec["num_q_heads"] // Hkv * W
    k_read = sum(N_L * Hkv * L * d * 2 for L in seq)
    gather = sum(Hkv * 2 * ((min(layer_budgets[l], L - W) + W) + (B + W)) * d * 2
                 for L in seq for l in range(N_L))
    secondary = sum(N_L * Hkv * (n * d * 2 + 8 * L) for L in seq)
    return k_read, gather, secondary


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

    def __init__(self, spec, sample, workers, sample_len, lam):
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
        meta = (sample_len, spec["window"], G, spec["budget"], lam[0], lam[1])
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
    """(q_bits, k_bits) of the first n_units units (layer-major, then KV head) of
    request 0, generated on the CPU."""
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


def _layer0_lambdas(spec):
    from oracle import kv_evict_oracle as O
    from paper_2609_30738_gb300.workloads import lambda_arrays
    l1, l2 = lambda_arrays(spec, O.depth_profile)
    return float(l1[0]), float(l2[0])


def run_reference(args):
    """--impl reference: the fp64 oracle on the host cores. A step is one pass over a
    bounded sample (one unit per host core) of request 0 of the workload; the line
    reports the measured wall time of that pass as ms_per_step and the throughput
    of the sample (its share of the request's prefix tokens per second)."""
    world, rank, _ = _dist()
    if rank != 0:
        return
    from paper_2609_30738_gb300.workloads import WORKLOADS
    name = args.workload
    spec = WORKLOADS[name]
    cores = os.cpu_count() or 1
    n_units = cores          # one unit per host core and step
    L = spec["seq_lens"][0]
    sample = _oracle_sample_from_host(spec, n_units, 2609)
    pool = OraclePool(spec, sample, cores, L, _layer0_lambdas(spec))
    try:
        for _ in range(args.warmup):
            pool.run()
        times = [pool.run() for _ in range(args.steps)]
    finally:
        pool.close()
    step_s = sum(times) / len(times)
    units_req = spec["num_layers"] * spec["num_kv_heads"]
    tok_s = L * (n_units / units_req) / step_s
    desc = (f"{n_units} of the {units_req} units of request 0 (L = {L}; score + select, one unit "
            f"per worker) per step; measured wall {step_s * 1e3:.1f} ms per step")
    line = {"impl": "reference", "metric": METRIC, "value": tok_s, "unit": "prefix tok/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": step_s * 1e3, "higher_is_better": True,
            "scaling": "weak" if len(spec["seq_lens"]) == 1 else "strong",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded Mistral-7B-shaped K/Q)",
            "config": _config(name, spec, world),
            "sample_units_per_step": n_units,
            "extrapolated_ms_per_request": step_s * 1e3 * units_req / n_units,
            "cpu_baseline": {"value": tok_s, "unit": "prefix tok/s", "cores": cores, "kind": "oracle",
                             "sample": desc},
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
    name = args.workload
    full = WORKLOADS[name]
    reqs, scaling = _rank_requests(full, world, rank)
    spec = dict(full, seq_lens=[full["seq_lens"][0]] * len(reqs) if len(full["seq_lens"]) == 1
                else [full["seq_lens"][r] for r in reqs])
    if args.layers:
        spec = dict(spec, num_layers=args.layers)
    W, B, d = spec["window"], spec["budget"], spec["head_dim"]
    N_L, Hkv = spec["num_layers"], spec["num_kv_heads"]
    seq = spec["seq_lens"]
    tokens = sum(seq)                      # prefix tokens this rank evicts per step
    # requests per step over the job (weak: one per rank; strong: the batch)
    job_requests = world if scaling == "weak" else len(full["seq_lens"])

    # inputs resident in HBM; a batch's subset keeps its requests' seeds
    batch = synth.make_batch(spec, seed=2609, device=dev, request_ids=reqs) if reqs else None
    lam1, lam2 = lambda_arrays(spec, K.profile)
    stream = torch.cuda.Stream(device=dev)
    if batch is not None:
        q, k, v = batch["q_win"], batch["k"], batch["v"]
        plan = K.Plan(spec, batch["seq_lens"])
        bufs = K.Buffers(plan, device=dev, with_trace=False)

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

    # no garbage collection while GPU work is being enqueued: a collection pause of the
    # host thread (tens of ms with torch loaded) would leave the GPU idle inside a timed
    # region; collected once here and re-enabled after the last timed region
    gc.collect()
    gc.disable()
    sampler = ClockSampler(local) if rank == 0 else None
    if sampler:
        sampler.start()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    if sampler:
        sampler.mark("t0")
    t0.record(stream)
    # no event between the launches: the selection (with the compact cache) starts as a
    # programmatic dependent of the score kernel, which an event record in between would
    # prevent
    for i in range(args.steps if batch is not None else 0):
        plan.score(q, k, bufs.mu, bufs.sigma, bufs.ws, stream)
        plan.select_gather(bufs.mu, bufs.sigma, k, v, lam1, lam2, bufs.indices, bufs.k_out, bufs.v_out,
                           bufs.ws, None, None, stream)
    t1.record(stream)
    torch.cuda.synchronize()
    if sampler:
        sampler.mark("t1")
    if world > 1:
        dist.barrier()
    elapsed = t0.elapsed_time(t1) / 1e3
    # the dominant kernel's launch duration for the roofline: the same number of steps
    # right after the timed region, an event pair around each score launch on the bench
    # stream (the selection still runs between them)
    score_s = 0.0
    if batch is not None:
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(args.steps)]
        for i in range(args.steps):
            ev[i][0].record(stream)
            plan.score(q, k, bufs.mu, bufs.sigma, bufs.ws, stream)
            ev[i][1].record(stream)
            plan.select_gather(bufs.mu, bufs.sigma, k, v, lam1, lam2, bufs.indices, bufs.k_out,
                               bufs.v_out, bufs.ws, None, None, stream)
        torch.cuda.synchronize()
        score_s = sum(a.elapsed_time(b) for a, b in ev) / 1e3 / args.steps
    clocks = sampler.stop() if sampler else None
    if batch is not None and plan.status(bufs.ws, stream) != K.KVE_OK:
        raise RuntimeError("device-side wait timed out in the timed region")
    elapsed = _max_over_ranks(elapsed, world, dev)

    # the score pass with the window rows' attention output (kv_evict_score_attn): the
    # same K stream plus V, timed alone beside the plain score kernel
    window = None
    if batch is not None and args.attn_steps > 0:
        attn_ws = torch.empty(plan.score_attn_workspace(), dtype=torch.uint8, device=dev)
        o_win = torch.empty_like(q)
        with torch.cuda.stream(stream):
            plan.score_attn(q, k, v, bufs.mu, bufs.sigma, o_win, bufs.ws, attn_ws, stream)
        if plan.status(bufs.ws, stream) != K.KVE_OK:
            raise RuntimeError("device-side wait timed out in the window-output pass")
        wa, wb = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        wa.record(stream)
        for _ in range(args.attn_steps):
            plan.score_attn(q, k, v, bufs.mu, bufs.sigma, o_win, bufs.ws, attn_ws, stream)
        wb.record(stream)
        torch.cuda.synchronize()
        attn_s = wa.elapsed_time(wb) / 1e3 / args.attn_steps
        kv_bytes = 2 * sum(N_L * Hkv * Lr * d * 2 for Lr in seq)
        window = {"score_attn_ms": attn_s * 1e3, "score_ms": score_s * 1e3,
                  "kv_read_bytes": kv_bytes, "kv_read_gbs": kv_bytes / attn_s / 1e9,
                  "attn_ws_bytes": int(attn_ws.numel())}
        del attn_ws, o_win

    # the score pass given the window rows' softmax normalisers (kv_evict_score_lse: a
    # prefill's attention has them), timed alone beside the two-pass score kernel; the
    # normalisers come from a float32 computation of the window logits (set-up, untimed)
    given_lse = None
    if batch is not None and args.lse_steps > 0:
        lse = _window_lse(spec, batch, dev)
        with torch.cuda.stream(stream):
            plan.score_lse(q, k, lse, bufs.mu, bufs.sigma, bufs.ws, stream)
        if plan.status(bufs.ws, stream) != K.KVE_OK:
            raise RuntimeError("device-side wait timed out in the given-normaliser pass")
        la, lb = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        la.record(stream)
        for _ in range(args.lse_steps):
            plan.score_lse(q, k, lse, bufs.mu, bufs.sigma, bufs.ws, stream)
        lb.record(stream)
        torch.cuda.synchronize()
        lse_s = la.elapsed_time(lb) / 1e3 / args.lse_steps
        # and the whole step in that form: the given-normaliser score, then the selection
        # with the compact cache
        la.record(stream)
        for _ in range(args.lse_steps):
            plan.score_lse(q, k, lse, bufs.mu, bufs.sigma, bufs.ws, stream)
            plan.select_gather(bufs.mu, bufs.sigma, k, v, lam1, lam2, bufs.indices, bufs.k_out,
                               bufs.v_out, bufs.ws, None, None, stream)
        lb.record(stream)
        torch.cuda.synchronize()
        lstep_s = la.elapsed_time(lb) / 1e3 / args.lse_steps
        k_bytes = sum(N_L * Hkv * Lr * d * 2 for Lr in seq)
        given_lse = {"score_lse_ms": lse_s * 1e3, "score_ms": score_s * 1e3, "k_read_bytes": k_bytes,
                     "k_read_gbs": k_bytes / lse_s / 1e9, "frac_of_peak": k_bytes / lse_s / 1e9 / _peaks()[0],
                     "step_ms": lstep_s * 1e3,
                     "step_frac_of_peak": sum(_algorithmic_bytes(spec, seq, plan.layer_budgets)[:2])
                     / lstep_s / 1e9 / _peaks()[0],
                     "note": "lse is an input here (a prefill's attention computes it); not the headline step"}
        del lse

    # end to end through the public API with host buffers (pinned), copies inside.
    # A one-request call is evicted in chunks of layers, one plan per chunk: the copy
    # stream brings in chunk c + 1 while the compute stream scores, selects and
    # gathers chunk c (every array is layer-major for one request, so a chunk is a
    # contiguous view). V stays in pinned host memory: the selection's compact-cache
    # write reads the kept rows in place, so min(B_l, L_r - W) + W rows per unit cross
    # the host link, not the whole tensor.
    e2e = None
    if args.e2e_steps > 0:
        e2e_s, h2d, d2h, chunks, steps_ms = 0.0, 0, 0, 1, []
        if batch is not None:
            e2e_s, h2d, d2h, chunks, steps_ms = _e2e(args, spec, batch, plan, bufs, lam1, lam2, stream,
                                                     dev, world)
        elif world > 1:
            dist.barrier()                 # the one in _e2e, for a rank without requests
        e2e_s = _max_over_ranks(e2e_s, world, dev)
        job_tokens = tokens * world if scaling == "weak" else sum(full["seq_lens"])
        e2e = {"value": job_tokens / e2e_s, "unit": "prefix tok/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": e2e_s * 1e3, "layer_chunks": chunks,
               "step_ms_min_max": [min(steps_ms), max(steps_ms)] if steps_ms else None,
               "step_ms_median": sorted(steps_ms)[len(steps_ms) // 2] if steps_ms else None,
               "step_ms": [round(x, 3) for x in steps_ms],
               "v": "read in place from pinned host memory by the compact-cache write (kept rows only)"}

    gc.enable()
    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return

    # roofline: algorithmic bytes (K read + K/V gathered) over the measured HBM peak;
    # the dominant kernel (score) reads K
    k_read, gather_bytes, secondary = _algorithmic_bytes(spec, seq, plan.layer_budgets)
    peak, peak_kind = _peaks()
    achieved = k_read / score_s / 1e9
    traffic = (SCORE_TRAFFIC["bytes_per_launch"]
               if (SCORE_TRAFFIC["source_sha256"] == _score_source_sha() and name == WORKLOAD
                   and not args.layers) else None)

    cpu = None
    if world == 1 and args.cpu_units > 0:
        cpu = cpu_baseline_from_device(spec, batch, args.cpu_units)

    step_s = elapsed / args.steps
    job_tokens = tokens * world if scaling == "weak" else sum(full["seq_lens"])
    config = _config(name, full, world)
    if args.layers:
        config["workload"] = f"{name} ({N_L} layers)"
    line = {"metric": METRIC, "value": job_tokens / step_s, "unit": "prefix tok/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": step_s * 1e3,
            "higher_is_better": True, "scaling": scaling, "vs_baseline": None,
            "dtype": "bf16xbf16->f32", "data": "synthetic (seeded Mistral-7B-shaped K/V/Q)",
            "config": config,
            "ms_per_request": step_s * 1e3 * world / job_requests,
            "hbm_roofline_frac_step": (k_read + gather_bytes) / step_s / 1e9 / peak,
            "algorithmic_bytes_step": {"k_read": k_read, "kv_gathered": gather_bytes},
            "score_kernel_ms": score_s * 1e3,
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak, "traffic": traffic,
                         "peak_source": peak_kind, "kernel": "kve score_kernel",
                         "algorithmic_bytes_per_launch": k_read,
                         "secondary_bytes_per_launch": secondary},
            "gpu_launches": 2 * args.steps,
            "clocks": clocks, "cpu_baseline": cpu, "e2e": e2e, "window_output": window,
            "given_lse": given_lse}
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def _window_lse(spec, batch, dev):
    """Natural-log softmax normaliser of every window row, [N_L][n_req][Hq][W] fp32 in q_win's
    row order, from a float32 computation of the window logits (TF32 off): the input of
    kv_evict_score_lse, as a prefill attention would hand it over."""
    import torch
    N_L, Hq, Hkv, W, d = (spec[x] for x in ("num_layers", "num_q_heads", "num_kv_heads", "window", "head_dim"))
    G = Hq // Hkv
    q, k, seq = batch["q_win"], batch["k"], batch["seq_lens"]
    out = torch.empty((N_L, len(seq), Hq, W), dtype=torch.float32, device=dev)
    prev = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = False
    try:
        off = 0
        for r, L in enumerate(seq):
            vis = torch.arange(L, device=dev)[None, :] <= torch.arange(L - W, L, device=dev)[:, None]
            for layer in range(N_L):
                for h in range(Hkv):
                    qq = q[layer, r, h * G:(h + 1) * G].float()
                    lg = torch.einsum("gwd,ld->gwl", qq, k[layer, h, off:off + L].float()) / math.sqrt(d)
                    out[layer, r, h * G:(h + 1) * G] = torch.logsumexp(lg.masked_fill(~vis, -math.inf), dim=-1)
            off += L
    finally:
        torch.backends.cuda.matmul.allow_tf32 = prev
    return out


def _e2e(args, spec, batch, plan, bufs, lam1, lam2, stream, dev, world):
    """End-to-end step through the public API: seconds per step, H2D and D2H bytes
    per step, layer chunks."""
    import torch
    import torch.distributed as dist
    from paper_2609_30738_gb300 import kv_evict as K
    q, k, v = batch["q_win"], batch["k"], batch["v"]
    W, d = spec["window"], spec["head_dim"]
    N_L, Hkv = spec["num_layers"], spec["num_kv_heads"]
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
    idx_c = bufs.indices.view(chunks, -1, bufs.indices.shape[1])
    ko_c = bufs.k_out.view(chunks, -1, *bufs.k_out.shape[1:])
    vo_c = bufs.v_out.view(chunks, -1, *bufs.v_out.shape[1:])
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
            cplan.select_gather(mu_c[c], sg_c[c], dk[ls], hv[ls], lam1[ls], lam2[ls], idx_c[c], ko_c[c],
                                vo_c[c], cws, None, None, stream)
        with torch.cuda.stream(stream):
            o_idx.copy_(bufs.indices, non_blocking=True)
            o_k.copy_(bufs.k_out, non_blocking=True)
            o_v.copy_(bufs.v_out, non_blocking=True)

    for _ in range(3):                     # first touches of the pinned buffers
        e2e_step()
    stream.synchronize()
    if cplan.status(cws, stream) != K.KVE_OK:
        raise RuntimeError("device-side wait timed out in the end-to-end step")
    # an event at every step boundary (each step's copies wait for the previous step, so
    # consecutive events bracket one step): the mean over the steps is the measurement,
    # the spread is reported beside it
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.e2e_steps + 1)]
    if world > 1:
        dist.barrier()
    copy_stream.wait_stream(stream)
    ev[0].record(copy_stream)
    for i in range(args.e2e_steps):
        e2e_step()
        ev[i + 1].record(stream)
    torch.cuda.synchronize()
    if cplan.status(cws, stream) != K.KVE_OK:
        raise RuntimeError("device-side wait timed out in the end-to-end step")
    e2e_s = ev[0].elapsed_time(ev[-1]) / 1e3 / args.e2e_steps
    steps_ms = [ev[i].elapsed_time(ev[i + 1]) for i in range(args.e2e_steps)]
    h2d = sum(x.numel() * x.element_size() for x in (hq, hk)) + v_read
    d2h = sum(x.numel() * x.element_size() for x in (o_idx, o_k, o_v))
    return e2e_s, h2d, d2h, chunks, steps_ms


def cpu_baseline_from_device(spec, batch, n_units):
    """Oracle on the first n_units units (request 0) of the device-resident inputs:
    the measured wall time of that sample, and the throughput it implies."""
    from tests.parity import to_bits
    G = spec["num_q_heads"] // spec["num_kv_heads"]
    W, Hkv, L = spec["window"], spec["num_kv_heads"], spec["seq_lens"][0]
    units_req = spec["num_layers"] * Hkv
    n_units = min(n_units, units_req)
    sample = []
    for u in range(n_units):
        layer, h = divmod(u, Hkv)
        sample.append((to_bits(batch["q_win"][layer, 0, h * G:(h + 1) * G]).reshape(G * W, -1),
                       to_bits(batch["k"][layer, h, :L])))
    cores = min(os.cpu_count() or 1, n_units)
    pool = OraclePool(spec, sample, cores, L, _layer0_lambdas(spec))
    try:
        wall = pool.run()
    finally:
        pool.close()
    return {"value": L * (n_units / units_req) / wall, "unit": "prefix tok/s", "cores": cores,
            "kind": "oracle",
            "sample": f"{n_units} of the {units_req} units of request 0 (L = {L}; score + select) "
                      f"on {cores} worker processes",
            "sample_wall_s": wall,
            "extrapolated_ms_per_request": wall * 1e3 * units_req / n_units}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=500)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=BENCH_WORKLOADS, default=WORKLOAD)
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--e2e-chunks", type=int, default=8,
                    help="layer chunks of the end-to-end step (copy of chunk c+1 beside compute of c)")
    ap.add_argument("--cpu-units", type=int, default=128)
    ap.add_argument("--attn-steps", type=int, default=10,
                    help="launches of the score pass with the window output, timed beside the step")
    ap.add_argument("--lse-steps", type=int, default=10,
                    help="launches of the score pass given the window rows' normalisers, timed beside the step")
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
