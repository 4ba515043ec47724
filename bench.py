#!/usr/bin/env python3
"""Benchmark of the batched routing path on the config-4 burst workload.

One step = one smetric_route_batch call over one batch of 8,192 requests
(block hash, session key, two-tier prefix match, cost, argmin). Inputs are
resident in HBM when the timed region starts; four distinct batches of
~820 MB each rotate, so every step reads inputs larger than L2.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

With N > 1 the script runs under torchrun, one rank per GPU: every rank holds
a replica of the (static) index and routes its own batches; there is no
collective on the data path (weak scaling). Rank 0 prints one JSON line.
--impl reference times the CPU oracle on the host cores instead.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "routed requests/sec and prompt tokens hashed+matched/sec on 1 GB300; % HBM roofline"
UNIT = "requests/s"
WORKLOAD = ("c4_burst: 65536 concurrent sessions, Zipf(1.1) popularity, 64 instances, block 32, "
            "prompts U[8k,40k] tokens with a 95% cached prefix, index pre-populated at load "
            "factor 0.7, batches of 8192 requests")
N_DISTINCT_BATCHES = 4
NOMINAL_HBM_GBS = 7900.0  # GB300's nominal HBM3e bandwidth (context beside the measured copy peak)


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--e2e-steps", type=int, default=8)
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="target CPU time of the oracle baseline sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--sessions", type=int, default=65536,
                    help="sessions of the burst workload (smaller values: profiling cases)")
    ap.add_argument("--batch", type=int, default=8192, help="requests per batch")
    ap.add_argument("--sweep", action="store_true",
                    help="config-5 stress sweep instead of the benchmark line: batch, N and B "
                         "varied on the config-4 generator, table filled to --table-gb")
    ap.add_argument("--table-gb", type=float, default=40.0)
    ap.add_argument("--commit", action="store_true",
                    help="time device-side index maintenance (route, then commit the batch's blocks "
                         "and drain the queues) over a config-2 replay (one GPU; its own JSON line)")
    ap.add_argument("--sequential", action="store_true",
                    help="time the sequential-update variant on the config-4 workload (one GPU; its own line)")
    ap.add_argument("--link", action="store_true",
                    help="time session reconstruction (Appendix A) over a config-3 trace (one GPU; its own line)")
    ap.add_argument("--reuse", action="store_true",
                    help="time the KV$ reuse breakdown (Section 3.1) over a whole config-2 window "
                         "(one GPU; its own line)")
    ap.add_argument("--pipeline", action="store_true",
                    help="time smetric_route_batches (the config-4 batches routed four per call, "
                         "alternating between two scratch sets) against one smetric_route_batch per batch")
    ap.add_argument("--imbalance", action="store_true",
                    help="time the windowed load imbalance (Section 3.2) over a day of running intervals "
                         "(one GPU; its own line)")
    ap.add_argument("--coloc", action="store_true",
                    help="with --policy: the PD-colocation variant (Appendix B)")
    ap.add_argument("--policy", action="store_true",
                    help="time the session-centric policy (Figure 10) instead of the argmin cost "
                         "(one GPU; its own JSON line)")
    return ap.parse_args()


def dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist  # noqa: F811
        backend = "nccl" if args.impl == "ours" else "gloo"
        if backend == "nccl":
            import torch
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return rank, world, local, dist


# ---------------------------------------------------------------------------
# clocks
# ---------------------------------------------------------------------------

class ClockSampler:
    """nvidia-smi samples of SM clock, power and throttle reasons."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu: str):
        self.gpu = gpu
        self.proc = None
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        self.t0 = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", str(self.gpu)], stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        self.t0 = time.time()

    def n_samples(self) -> int:
        """Rows written so far."""
        try:
            with open(self.f.name) as g:
                return sum(1 for r in g if r.strip())
        except OSError:
            return 0

    def soak(self, step, min_samples=8, max_seconds=6.0):
        """Runs `step(i)` (untimed, synchronising every 50 calls) until the
        sampler holds at least `min_samples` rows or `max_seconds` pass, so
        that a short timed region still gets a clock record of the same load
        around it. Returns the number of steps run."""
        import torch
        if self.proc is None:
            return 0
        t0, i = time.time(), 0
        while self.n_samples() < min_samples and time.time() - t0 < max_seconds:
            for _ in range(50):
                step(i)
                i += 1
            torch.cuda.synchronize()
        return i

    def stop(self, window="warm-up and timed steps"):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        self.f.flush()
        self.f.seek(0)
        rows = [r.split(", ") for r in self.f.read().strip().splitlines() if r.strip()]
        os.unlink(self.f.name)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            try:
                sm.append(float(r[1]))
                mx.append(float(r[2]))
                for n, v in zip(names, r[5:9]):
                    if v.strip().lower() == "active":
                        reasons.add(n)
            except (IndexError, ValueError):
                continue
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm),
                "window": window}


def h2d_link_gbs(pinned, device, reps=5):
    """Host-to-device copy rate of one pinned buffer (GB/s): the ceiling of
    the end-to-end number, which must move the batch's tokens every step."""
    import torch
    dst = torch.empty(pinned.numel(), dtype=pinned.dtype, device=device)
    dst.copy_(pinned, non_blocking=True)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        dst.copy_(pinned, non_blocking=True)
    e1.record()
    torch.cuda.synchronize()
    gbs = reps * pinned.numel() * pinned.element_size() / (e0.elapsed_time(e1) / 1e3) / 1e9
    del dst
    return gbs


def peak_hbm():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback"


def section_sha(section: str) -> str:
    """Hash of one kernel's source: its section of route.cu (from its
    `// <section>` banner to the next banner), the file's preamble of launch
    constants, and the shared device header, comments left out."""
    csrc = os.path.join(ROOT, "paper_2607_08565_gb300", "csrc")
    text = open(os.path.join(csrc, "route.cu")).read()
    banner = "// " + "-" * 75 + "\n"
    parts = text.split(banner)
    body = next((parts[i + 1] for i in range(len(parts) - 1) if parts[i].rstrip("\n").endswith("// " + section)), None)
    if body is None:
        return ""
    def code(t):  # comments and blank lines do not change a kernel
        out = []
        for line in t.splitlines():
            line = line.split("//")[0].rstrip()
            if line:
                out.append(line)
        return "\n".join(out).encode()

    h = hashlib.sha256(code(parts[0]) + code(body))
    h.update(code(open(os.path.join(csrc, "smetric_impl.cuh")).read()))
    return h.hexdigest()[:16]


def ncu_traffic(kernel: str):
    """Per-launch DRAM bytes of `kernel` from the committed ncu summary, if
    that summary was taken on the current kernel source; else None."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)[kernel]
    except (OSError, KeyError, ValueError):
        return None
    sha = section_sha(rec["section"]) if "section" in rec else ""
    return rec["bytes_per_launch"] if sha and sha == rec["source_sha"] else None


# ---------------------------------------------------------------------------
# workload
# ---------------------------------------------------------------------------

def c4_trace(args=None):
    from synth import burst_trace
    if args is None:
        return burst_trace()
    return burst_trace(n_sessions=args.sessions, batch_size=args.batch)


def workload_name(args):
    if args.sessions == 65536 and args.batch == 8192:
        return WORKLOAD
    return (f"c4_burst generator reduced to {args.sessions} sessions and batches of "
            f"{args.batch} requests (a profiling case, not the benchmark workload)")


def populate_index(ix, tr, device, chunk=4096):
    import torch
    B = tr.params.block_size
    buf = np.empty(int(tr.prefix_len.max()) * chunk, np.int32)
    for ids, tok, off in tr.prepopulation(chunk=chunk, out=buf):
        hb, _ = ix.block_hashes(torch.from_numpy(tok).to(device), torch.from_numpy(off).to(device))
        nb = torch.from_numpy(tr.prefix_len[ids] // B).to(device)
        hb = hb[:int(nb.sum())].view(torch.int64)  # CUDA mask indexing has no uint64 kernels
        owner = torch.repeat_interleave(torch.arange(len(ids), device=device), nb)
        sess = torch.from_numpy(ids).to(device)[owner]
        ix.insert(hb, -1)
        for tier_of, member in ((tr.home, tr.in_home), (tr.second, tr.in_second)):
            m = torch.from_numpy(member).to(device)[sess]
            t = torch.from_numpy(tier_of).to(device)[sess]
            ix.insert(hb[m].contiguous(), t[m].contiguous())
    ix.check()


def algorithmic_bytes(lens, local_hit, global_hit, B, W):
    """Per-kernel bytes of one route call. k_digest: 4 B per hashed token (the
    method must read every token of every full block). k_probe: one index
    entry (key + W mask words) per probed block, P_r = min(n_r, reach_r + 1),
    with reach_r taken from the chosen instance's hits, g_{i*} = max(c_{i*}, g):
    never above max(max_i c_i, g), and equal to it when the global tier holds
    every local tier's blocks (config 4), so the count never overstates.
    k_chain_probe adds to those entries the digests the chain reads and the
    hashes it writes (8 B each per block). k_walk: the masks it reads, offsets
    and outputs. k_prep: offsets and loads. path: the method's bytes per
    request, 4 L_r + P_r (8 + 8W) + 8 + 20."""
    nb = lens // B
    reach = (local_hit.astype(np.int64) + global_hit) // B
    probes = np.minimum(nb, reach + 1)
    n = len(lens)
    return {
        "k_digest": int(4 * B * nb.sum()),
        "k_probe": int(probes.sum() * (8 + 8 * W)),
        "k_chain_probe": int(16 * nb.sum() + 24 * n + probes.sum() * (8 + 8 * W)),
        "k_walk": int(8 * W * probes.sum() + 28 * n),
        "k_prep": int(16 * n),
        "path": int(4 * lens.sum() + probes.sum() * (8 + 8 * W) + 8 * (n + 1) + 20 * n),
    }


def route_stats(lens_per_batch, outs_per_batch, num_instances):
    """Serving-side view of the routed batches (the paper's reuse and
    imbalance metrics, Sections 3.1-3.2, taken from the route's outputs):
    the share of prompt tokens hit in the chosen instance's local tier and
    fetched from the global tier, and the routed-token imbalance of each
    batch, N * max_i (tokens routed to i) / (all tokens), averaged over the
    batches."""
    tok = loc = glob = 0
    imb = []
    for lens, o in zip(lens_per_batch, outs_per_batch):
        lens = np.asarray(lens, np.int64)
        tok += int(lens.sum())
        loc += int(np.asarray(o["local_hit"], np.int64).sum())
        glob += int(np.asarray(o["global_hit"], np.int64).sum())
        per = np.bincount(np.asarray(o["instance"], np.int64), weights=lens, minlength=num_instances)
        if per.sum() > 0:
            imb.append(float(num_instances * per.max() / per.sum()))
    return {"local_hit_ratio": loc / tok if tok else 0.0,
            "global_hit_ratio": glob / tok if tok else 0.0,
            "routed_token_imbalance": float(np.mean(imb)) if imb else None,
            "batches": len(imb)}


# ---------------------------------------------------------------------------
# CPU oracle timing
# ---------------------------------------------------------------------------

def oracle_index_for(tr, batches):
    """Oracle index holding every session prefix the given batches use."""
    import oracle
    p = tr.params
    ox = oracle.OracleIndex(p.num_instances)
    sessions = np.unique(np.concatenate([b.sessions for b in batches]))
    for s in sessions.tolist():
        h = oracle.block_hashes(tr.session_prefix(s), p.block_size, p.hash_seed)
        for t in tr.session_tiers(s):
            ox.insert(h, t)
    return ox


def oracle_route(tr, ox, bt, m, threads):
    """Seconds the oracle takes to route the first m requests of bt."""
    p = tr.params
    off = bt.offsets[:m + 1]
    t0 = time.perf_counter()
    ox.route_batch(p.block_size, p.session_blocks, p.hash_seed, bt.tokens[:off[-1]], off,
                   bt.load, p.w_load, p.w_miss, p.w_glob, n_threads=threads)
    return time.perf_counter() - t0


def oracle_calibrate(tr, ox, bt, seconds, threads):
    """Largest prefix m of the batch (doubling from 64) routed in about
    `seconds`; returns (m, seconds taken)."""
    m = min(64, bt.n_requests)
    while True:
        dt = oracle_route(tr, ox, bt, m, threads)
        if dt >= seconds / 2 or m == bt.n_requests:
            return m, dt
        m = min(bt.n_requests, max(m * 2, int(m * seconds / max(dt, 1e-3))))


def cpu_baseline(tr, bt, batch_id, seconds, threads=None):
    """The oracle timed on the host cores on batch `bt`: a bounded sample of
    about `seconds` on every core (the whole batch repeated when it is
    quicker), and a smaller sample on one thread."""
    threads = threads or os.cpu_count() or 1
    ox = oracle_index_for(tr, [bt])
    m, dt = oracle_calibrate(tr, ox, bt, seconds, threads)
    reps = 1
    if m == bt.n_requests and dt < seconds / 2:
        # the whole batch is quicker than the target: route it repeatedly
        reps = max(2, int(seconds / max(dt, 1e-3)))
        t0 = time.perf_counter()
        for _ in range(reps):
            oracle_route(tr, ox, bt, m, threads)
        dt = time.perf_counter() - t0
    what = (f"{reps} passes over all {m} requests" if reps > 1 else
            f"first {m} of the {bt.n_requests} requests")
    m1, dt1 = oracle_calibrate(tr, ox, bt, seconds / 4, 1)
    ox.close()
    return {"value": reps * m / dt, "unit": UNIT, "cores": threads, "kind": "oracle",
            "sample": f"{what} of config-4 batch {batch_id} ({dt:.1f} s on {threads} threads), "
                      f"oracle index holding that batch's sessions",
            "tokens_per_s": reps * float(bt.offsets[m]) / dt,
            "single_thread": {"value": m1 / dt1, "unit": UNIT, "cores": 1,
                              "sample": f"first {m1} requests of the same batch ({dt1:.1f} s on one thread)"}}


def run_reference(args, rank, world, dist):
    if rank != 0:
        return
    import oracle
    oracle.build()
    tr = c4_trace(args)
    threads = os.cpu_count() or 1
    batches = [tr.batch(k) for k in range(N_DISTINCT_BATCHES)]
    ox = oracle_index_for(tr, batches)
    per_step = min(2.0, 150.0 / max(1, args.warmup + args.steps))
    m, _ = oracle_calibrate(tr, ox, batches[0], per_step, threads)
    for i in range(args.warmup):
        oracle_route(tr, ox, batches[i % len(batches)], m, threads)
    times, toks = [], 0
    for i in range(args.steps):
        bt = batches[i % len(batches)]
        times.append(oracle_route(tr, ox, bt, m, threads))
        toks += int(bt.offsets[m])
    total = sum(times)
    rps = args.steps * m / total
    sample = (f"first {m} of the {batches[0].n_requests} requests of a config-4 batch per step "
              f"(4 batches rotated), "
              f"oracle index holding those batches' sessions, {threads} threads")
    line = {
        "impl": "reference", "metric": METRIC, "value": rps, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u64",
        "data": "synthetic", "tokens_per_s": toks / total,
        "config": {"workload": workload_name(args), "l2": "host run"},
        "cpu_baseline": {"value": rps, "unit": UNIT, "cores": threads, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": rps, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------

def run_ours(args, rank, world, local, dist):
    import torch
    import paper_2607_08565_gb300 as pkg
    from paper_2607_08565_gb300 import build_lib

    if rank == 0 or not build_lib.up_to_date():
        build_lib.build()
    if dist is not None:
        dist.barrier()
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    tr = c4_trace(args)
    p = tr.params
    N, B = p.num_instances, p.block_size

    # this rank's batches: ids rank, rank + world, ... (distinct across ranks)
    ids = [rank + world * i for i in range(N_DISTINCT_BATCHES)]
    host = [tr.batch(k) for k in ids]
    nkeys = tr.n_prefix_blocks()
    chunk = 4096  # sessions hashed per pre-population call
    max_tok = max(max(b.n_tokens for b in host), chunk * int(tr.prefix_len.max()))
    ix = pkg.SMetricIndex(N, B, p.session_blocks, capacity_slots=int(nkeys / 0.7) + 1,
                          max_batch_requests=max(tr.batch_size, chunk), max_batch_tokens=max_tok,
                          hash_seed=p.hash_seed, host_staging=True)
    populate_index(ix, tr, device, chunk)
    dev_b = []
    for b in host:
        dev_b.append(dict(tok=torch.from_numpy(b.tokens).to(device),
                          off=torch.from_numpy(b.offsets).to(device),
                          load=torch.from_numpy(b.load).to(device), n=b.n_requests,
                          n_tokens=b.n_tokens))
    n = tr.batch_size
    outs = dict(instance=torch.empty(n, dtype=torch.int32, device=device),
                local_hit=torch.empty(n, dtype=torch.int32, device=device),
                global_hit=torch.empty(n, dtype=torch.int32, device=device),
                session_key=torch.empty(n, dtype=torch.uint64, device=device))
    w = (p.w_load, p.w_miss, p.w_glob)
    stream = torch.cuda.current_stream(device)

    def step(i):
        b = dev_b[i % len(dev_b)]
        pkg.smetric_route_batch(ix.handle, b["tok"], b["n_tokens"], b["off"], b["n"], b["load"], w,
                                outs["instance"], outs["local_hit"], outs["global_hit"],
                                outs["session_key"], None, 0, stream)

    # per-batch outputs (for the algorithmic-byte count)
    per_batch = []
    for i in range(len(dev_b)):
        step(i)
        ix.check()
        per_batch.append({k: v.cpu().numpy().copy() for k, v in outs.items()})

    try:
        gpu_id = "GPU-" + str(torch.cuda.get_device_properties(local).uuid)
    except Exception:
        gpu_id = str(local)
    clocks = ClockSampler(gpu_id)
    clocks.start()
    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    launches0 = pkg.smetric_launch_count(ix.handle)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for i in range(args.steps):
        step(i)
    ev1.record(stream)
    torch.cuda.synchronize()
    ms = ev0.elapsed_time(ev1)
    launches = pkg.smetric_launch_count(ix.handle) - launches0
    soaked = clocks.soak(step)
    clk = clocks.stop("warm-up and timed steps" + (f", then {soaked} more of the same steps (untimed) so that "
                                                   f"the sampler, every 100 ms, records the load" if soaked else ""))
    rc = ix.status()
    if rc != pkg.SMETRIC_OK:
        raise pkg.SmetricError(rc, "bench")
    if dist is not None:
        t = torch.tensor([ms], device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
        if dist is not None:
            dist.barrier()

    reqs_per_step = np.mean([b.n_requests for b in host])
    toks_per_step = np.mean([b.n_tokens for b in host])
    value = world * args.steps * reqs_per_step / (ms / 1e3)
    tokens_per_s = world * args.steps * toks_per_step / (ms / 1e3)

    # per-kernel durations, measured live with CUDA events on the launch stream
    pkg.smetric_profile_enable(ix.handle, True)
    kprof_steps = max(20, min(args.steps, 200))
    for i in range(kprof_steps):
        step(i)
    prof = pkg.smetric_profile_read(ix.handle)
    pkg.smetric_profile_enable(ix.handle, False)
    algo = [algorithmic_bytes(b.lengths(), pb["local_hit"], pb["global_hit"], B, ix.W)
            for b, pb in zip(host, per_batch)]
    algo_mean = {k: float(np.mean([a[k] for a in algo])) for k in algo[0]}
    peak, peak_kind = peak_hbm()
    dom = max(prof, key=lambda k: prof[k][0])
    dom_ms = prof[dom][0] / max(prof[dom][1], 1)
    achieved = algo_mean[dom] / (dom_ms / 1e3) / 1e9
    path_ms = ms / args.steps
    path_gbs = algo_mean["path"] / (path_ms / 1e3) / 1e9
    traffic = ncu_traffic(dom)

    # end to end through the host-buffer entry point: H2D of the batch, route,
    # D2H of the outputs, every step
    pinned = []
    for b in host[:2]:
        t = torch.empty(b.n_tokens, dtype=torch.int32, pin_memory=True)
        t.numpy()[:] = b.tokens
        pinned.append(dict(tok=t, off=torch.from_numpy(b.offsets).pin_memory(),
                           load=torch.from_numpy(b.load).pin_memory(), n=b.n_requests,
                           n_tokens=b.n_tokens))
    hout = dict(instance=torch.empty(n, dtype=torch.int32, pin_memory=True),
                local_hit=torch.empty(n, dtype=torch.int32, pin_memory=True),
                global_hit=torch.empty(n, dtype=torch.int32, pin_memory=True),
                session_key=torch.empty(n, dtype=torch.uint64, pin_memory=True))

    def e2e_step(i):
        b = pinned[i % len(pinned)]
        rc = pkg.smetric_route_batch_host(ix.handle, b["tok"], b["n_tokens"], b["off"], b["n"],
                                          b["load"], w, hout["instance"], hout["local_hit"],
                                          hout["global_hit"], hout["session_key"], stream)
        if rc != pkg.SMETRIC_OK:
            raise pkg.SmetricError(rc, "e2e")

    for i in range(2):
        e2e_step(i)
    if dist is not None:
        dist.barrier()
    t0 = time.perf_counter()
    for i in range(args.e2e_steps):
        e2e_step(i)
    e2e_s = time.perf_counter() - t0
    if dist is not None:
        t = torch.tensor([e2e_s], device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        e2e_s = float(t.item())
    e2e_reqs = np.mean([b["n"] for b in pinned])
    e2e_value = world * args.e2e_steps * e2e_reqs / e2e_s
    h2d = float(np.mean([4 * b["n_tokens"] + 8 * (b["n"] + 1) + 8 * N for b in pinned]))
    d2h = float(20 * e2e_reqs)
    link = h2d_link_gbs(pinned[0]["tok"], device)
    # the host-buffer path must agree with the device path
    last = per_batch[(args.e2e_steps - 1) % len(pinned)]
    for k in hout:
        if not np.array_equal(hout[k].numpy(), last[k]):
            raise RuntimeError(f"host-buffer route differs from the device route in {k}")

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(tr, host[0], ids[0], args.cpu_seconds)

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": path_ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "u64", "data": "synthetic",
            "tokens_per_s": tokens_per_s,
            "config": {"workload": workload_name(args), "batch": int(reqs_per_step),
                       "num_instances": N, "block_size": B, "index_keys": nkeys,
                       "l2": f"inputs larger than L2: {N_DISTINCT_BATCHES} distinct batches of "
                             f"{toks_per_step * 4 / 1e6:.0f} MB rotated"},
            "roofline": {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": peak,
                         "unit": "GB/s", "frac": achieved / peak, "peak_kind": f"{peak_kind} copy",
                         "traffic": traffic, "algorithmic_bytes_per_launch": algo_mean[dom],
                         "ms_per_launch": dom_ms, "frac_of_nominal": achieved / NOMINAL_HBM_GBS},
            "roofline_path": {"achieved": path_gbs, "frac": path_gbs / peak,
                              "algorithmic_bytes_per_step": algo_mean["path"],
                              "frac_of_nominal": path_gbs / NOMINAL_HBM_GBS},
            "kernels_ms_per_launch": {k: v[0] / max(v[1], 1) for k, v in prof.items()},
            # every kernel against the same copy peak: the digest streams the
            # tokens (bound by its integer pipe at about this rate); the chain
            # and probe kernel is bound by the chain's dependent steps and
            # random entry reads, not by bandwidth
            "kernels_roofline": {k: {"achieved_gbs": algo_mean[k] / (v[0] / max(v[1], 1) / 1e3) / 1e9,
                                     "frac": algo_mean[k] / (v[0] / max(v[1], 1) / 1e3) / 1e9 / peak,
                                     "traffic": ncu_traffic(k)}
                                 for k, v in prof.items() if k in algo_mean and v[0] > 0},
            "route_stats": route_stats([b.lengths() for b in host], per_batch, N),
            "clocks": clk,
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h, "steps": args.e2e_steps,
                    "h2d_link_gbs": link,
                    "frac_of_link": (h2d * e2e_value / e2e_reqs / 1e9) / link if link else None},
            "gpu_launches": int(launches),
            "cpu_baseline": cpu,
        }
        print(json.dumps(line), flush=True)
    ix.close()
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()


# ---------------------------------------------------------------------------
# session-centric policy (Figure 10) on the same workload
# ---------------------------------------------------------------------------

# Eq. 1 in cost units: a 24k-token prompt with nothing cached costs ~3.1e8;
# queues are the batch's load draws (U[0, 2M]) scaled by 256, so up to 5.1e8;
# the TTFT deadline is 4e8 + 4,000 units per prompt token.
POLICY = dict(c_lin=1000, c_att=1, ttft_d0=400_000_000, ttft_d1=4000, hit_num=9, hit_den=10, rr_base=0)
QUEUED_SCALE = 256


def policy_inputs(tr, bt, k):
    """Per-request turn and expected hit, and per-instance queued cost, of
    batch k: a tenth of the requests open their session (turn 0), the others
    expect their session's cached prefix."""
    rng = np.random.default_rng([0x5E55_0005, k])
    turn = np.ones(bt.n_requests, np.int32)
    turn[rng.random(bt.n_requests) < 0.1] = 0
    est_hit = tr.prefix_len[bt.sessions].astype(np.int64)
    queued = bt.load.astype(np.int64) * QUEUED_SCALE
    return turn, est_hit, queued


def coloc_inputs(tr, k):
    """Per-instance TPOT budgets (a quarter of the instances run no decodes;
    the others absorb 1e7 to 1e9 cost units of prefill) and request counts
    (1 to 64) of batch k under PD colocation."""
    rng = np.random.default_rng([0x5E55_0006, k])
    N = tr.params.num_instances
    tpot = rng.integers(10 ** 7, 10 ** 9, size=N).astype(np.int64)
    tpot[rng.random(N) < 0.25] = 1 << 60
    return tpot, rng.integers(1, 65, size=N).astype(np.int64)


def run_policy(args):
    import torch
    import oracle
    import paper_2607_08565_gb300 as pkg
    from paper_2607_08565_gb300 import build_lib

    build_lib.build()
    torch.cuda.set_device(0)
    device = torch.device("cuda", 0)
    tr = c4_trace(args)
    p = tr.params
    N, B = p.num_instances, p.block_size
    ids = list(range(N_DISTINCT_BATCHES))
    host = [tr.batch(k) for k in ids]
    extra = [policy_inputs(tr, b, k) for b, k in zip(host, ids)]
    coloc = [coloc_inputs(tr, k) for k in ids] if args.coloc else None
    nkeys = tr.n_prefix_blocks()
    chunk = 4096
    max_tok = max(max(b.n_tokens for b in host), chunk * int(tr.prefix_len.max()))
    ix = pkg.SMetricIndex(N, B, p.session_blocks, capacity_slots=int(nkeys / 0.7) + 1,
                          max_batch_requests=max(tr.batch_size, chunk), max_batch_tokens=max_tok,
                          hash_seed=p.hash_seed)
    populate_index(ix, tr, device, chunk)
    T = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(device)
    dev_b = [dict(tok=T(b.tokens), off=T(b.offsets), n=b.n_requests, n_tokens=b.n_tokens, turn=T(tu),
                  est=T(eh), queued=T(q)) for b, (tu, eh, q) in zip(host, extra)]
    if coloc:
        for d, (tp, nr) in zip(dev_b, coloc):
            d["tpot"], d["nreq"] = T(tp), T(nr)
    n = tr.batch_size
    outs = dict(instance=torch.empty(n, dtype=torch.int32, device=device),
                local_hit=torch.empty(n, dtype=torch.int32, device=device),
                global_hit=torch.empty(n, dtype=torch.int32, device=device),
                stick=torch.empty(n, dtype=torch.int32, device=device),
                session_key=torch.empty(n, dtype=torch.uint64, device=device))
    stream = torch.cuda.current_stream(device)

    def step(i):
        b = dev_b[i % len(dev_b)]
        if coloc:
            pkg.smetric_route_batch_policy_coloc(ix.handle, b["tok"], b["n_tokens"], b["off"], b["n"],
                                                 b["queued"], b["tpot"], b["nreq"], b["turn"], b["est"], POLICY,
                                                 outs["instance"], outs["local_hit"], outs["global_hit"],
                                                 outs["stick"], outs["session_key"], None, 0, stream)
            return
        pkg.smetric_route_batch_policy(ix.handle, b["tok"], b["n_tokens"], b["off"], b["n"], b["queued"],
                                       b["turn"], b["est"], POLICY, outs["instance"], outs["local_hit"],
                                       outs["global_hit"], outs["stick"], outs["session_key"], None, 0,
                                       stream)

    per_batch = []
    for i in range(len(dev_b)):
        step(i)
        ix.check()
        per_batch.append({k: v.cpu().numpy().copy() for k, v in outs.items()})
    clocks = ClockSampler("GPU-" + str(torch.cuda.get_device_properties(0).uuid))
    clocks.start()
    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    launches0 = pkg.smetric_launch_count(ix.handle)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for i in range(args.steps):
        step(i)
    ev1.record(stream)
    torch.cuda.synchronize()
    ms = ev0.elapsed_time(ev1)
    launches = pkg.smetric_launch_count(ix.handle) - launches0
    soaked = clocks.soak(step)
    clk = clocks.stop("warm-up and timed steps" + (f", then {soaked} more of the same steps (untimed)"
                                                   if soaked else ""))
    if ix.status() != pkg.SMETRIC_OK:
        raise RuntimeError("policy bench: device error")
    reqs = float(np.mean([b.n_requests for b in host]))
    value = args.steps * reqs / (ms / 1e3)
    pkg.smetric_profile_enable(ix.handle, True)
    for i in range(max(20, min(args.steps, 200))):
        step(i)
    prof = pkg.smetric_profile_read(ix.handle)
    pkg.smetric_profile_enable(ix.handle, False)
    algo = [algorithmic_bytes(b.lengths(), pb["local_hit"], pb["global_hit"], B, ix.W)
            for b, pb in zip(host, per_batch)]
    algo_mean = {k: float(np.mean([a[k] for a in algo])) for k in algo[0]}
    peak, peak_kind = peak_hbm()
    dom = max(prof, key=lambda k: prof[k][0])
    dom_ms = prof[dom][0] / max(prof[dom][1], 1)
    achieved = algo_mean[dom] / (dom_ms / 1e3) / 1e9

    # end to end through the public API: pinned host inputs copied in, the
    # policy call, outputs read back, every step
    pin = lambda a: torch.from_numpy(np.ascontiguousarray(a)).pin_memory()
    hb = [dict(tok=pin(b.tokens), off=pin(b.offsets), turn=pin(tu), est=pin(eh), queued=pin(q), n=b.n_requests)
          for b, (tu, eh, q) in zip(host[:2], extra[:2])]
    stage = {k: torch.empty_like(v, device=device) for k, v in hb[0].items() if k != "n"}
    hout = {k: torch.empty(n, dtype=v.dtype, pin_memory=True) for k, v in outs.items()}

    if coloc:
        for d, (tp, nr) in zip(hb, coloc[:2]):
            d["tpot"], d["nreq"] = pin(tp), pin(nr)
        stage["tpot"] = torch.empty_like(hb[0]["tpot"], device=device)
        stage["nreq"] = torch.empty_like(hb[0]["nreq"], device=device)

    def e2e_step(i):
        b = hb[i % len(hb)]
        for k in ("tok", "off", "turn", "est", "queued") + (("tpot", "nreq") if coloc else ()):
            if stage[k].numel() < b[k].numel():
                stage[k] = torch.empty_like(b[k], device=device)
            stage[k][:b[k].numel()].copy_(b[k], non_blocking=True)
        if coloc:
            pkg.smetric_route_batch_policy_coloc(ix.handle, stage["tok"], b["tok"].numel(), stage["off"], b["n"],
                                                 stage["queued"], stage["tpot"], stage["nreq"], stage["turn"],
                                                 stage["est"], POLICY, outs["instance"], outs["local_hit"],
                                                 outs["global_hit"], outs["stick"], outs["session_key"], None, 0,
                                                 stream)
        else:
            pkg.smetric_route_batch_policy(ix.handle, stage["tok"], b["tok"].numel(), stage["off"], b["n"],
                                           stage["queued"], stage["turn"], stage["est"], POLICY, outs["instance"],
                                           outs["local_hit"], outs["global_hit"], outs["stick"],
                                           outs["session_key"], None, 0, stream)
        for k in hout:
            hout[k].copy_(outs[k], non_blocking=True)
        torch.cuda.synchronize()

    for i in range(2):
        e2e_step(i)
    t0 = time.perf_counter()
    for i in range(args.e2e_steps):
        e2e_step(i)
    e2e_s = time.perf_counter() - t0
    last = per_batch[(args.e2e_steps - 1) % len(hb)]
    for k in hout:
        if not np.array_equal(hout[k].numpy(), last[k]):
            raise RuntimeError(f"end-to-end policy route differs from the device route in {k}")
    h2d = float(np.mean([sum(b[k].numel() * b[k].element_size()
                             for k in ("tok", "off", "turn", "est", "queued") + (("tpot", "nreq") if coloc else ()))
                         for b in hb]))

    cpu = None
    if not args.no_cpu_baseline:
        ox = oracle_index_for(tr, host[:1])
        bt, (tu, eh, q) = host[0], extra[0]
        m, dt = 16, 0.0
        while True:  # the oracle's policy route runs on one thread
            off = bt.offsets[:m + 1]
            t0 = time.perf_counter()
            pv = [POLICY[k] for k in ("c_lin", "c_att", "ttft_d0", "ttft_d1", "hit_num", "hit_den", "rr_base")]
            if coloc:
                ox.route_batch_coloc(B, p.session_blocks, p.hash_seed, bt.tokens[:off[-1]], off, q, coloc[0][0],
                                     coloc[0][1], tu[:m], eh[:m], *pv)
            else:
                ox.route_batch_policy(B, p.session_blocks, p.hash_seed, bt.tokens[:off[-1]], off, q, tu[:m],
                                      eh[:m], *pv)
            dt = time.perf_counter() - t0
            if dt > args.cpu_seconds / 2 or m == bt.n_requests:
                break
            m = min(bt.n_requests, 2 * m)
        cpu = {"value": m / dt, "unit": UNIT, "cores": 1, "kind": "oracle",
               "sample": f"first {m} requests of config-4 batch 0 ({dt:.1f} s, one thread)"}

    stick = float(np.mean([pb["stick"].mean() for pb in per_batch]))
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": 1, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "u64", "data": "synthetic",
        "config": {"workload": workload_name(args), "batch": int(reqs), "num_instances": N, "block_size": B,
                   "decision": ("session-centric policy under PD colocation (Appendix B: TPOT filter, "
                                "LMetric product)" if coloc else
                                "session-centric policy (Figure 10, Eq. 1 in fixed point)"), "policy": POLICY,
                   "queued": f"batch load x {QUEUED_SCALE}", "first_turn_fraction": 0.1,
                   "stick_fraction": stick,
                   "l2": f"inputs larger than L2: {N_DISTINCT_BATCHES} distinct batches rotated"},
        "roofline": {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "peak_kind": f"{peak_kind} copy", "traffic": ncu_traffic(dom),
                     "algorithmic_bytes_per_launch": algo_mean[dom], "ms_per_launch": dom_ms},
        "kernels_ms_per_launch": {k: v[0] / max(v[1], 1) for k, v in prof.items()},
        "clocks": clk,
        "e2e": {"value": args.e2e_steps * reqs / e2e_s, "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": float(24 * reqs), "steps": args.e2e_steps},
        "gpu_launches": int(launches),
        "cpu_baseline": cpu,
    }
    print(json.dumps(line), flush=True)
    ix.close()


# ---------------------------------------------------------------------------
# sequential-update variant on the config-4 workload
# ---------------------------------------------------------------------------

def run_sequential(args, steps=50):
    import torch
    import paper_2607_08565_gb300 as pkg
    from paper_2607_08565_gb300 import build_lib

    build_lib.build()
    torch.cuda.set_device(0)
    tr = c4_trace(args)
    p = tr.params
    host = [tr.batch(k) for k in range(2)]
    nkeys = tr.n_prefix_blocks()
    chunk = 4096
    ix = pkg.SMetricIndex(p.num_instances, p.block_size, p.session_blocks, capacity_slots=int(nkeys / 0.7) + 1,
                          max_batch_requests=max(tr.batch_size, chunk),
                          max_batch_tokens=max(max(b.n_tokens for b in host), chunk * int(tr.prefix_len.max())),
                          hash_seed=p.hash_seed)
    populate_index(ix, tr, torch.device("cuda", 0), chunk)
    dev = [[torch.from_numpy(a).cuda() for a in (b.tokens, b.offsets, b.load)] for b in host]
    w = (p.w_load, p.w_miss, p.w_glob)
    times = {}
    for name, fn in (("snapshot", lambda d: ix.route_batch(*d, w)),
                     ("sequential", lambda d: ix.route_batch_sequential(*d, w))):
        for i in range(3):
            fn(dev[i % 2])
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for i in range(steps):
            out = fn(dev[i % 2])
        e1.record()
        torch.cuda.synchronize()
        ix.check()
        times[name] = e0.elapsed_time(e1) / steps
    seq = ix.route_batch_sequential(*dev[0], w)
    snap = ix.route_batch(*dev[0], w)
    changed = float((seq["instance"] != snap["instance"]).float().mean().item())
    line = {"metric": "routed requests/sec, loads updated request by request (sequential variant)",
            "value": host[0].n_requests / (times["sequential"] / 1e3), "unit": "requests/s", "n_gpus": 1,
            "steps": steps, "warmup": 3, "ms_per_step": times["sequential"], "snapshot_ms_per_step": times["snapshot"],
            "higher_is_better": True, "data": "synthetic",
            "config": {"workload": workload_name(args), "decisions_differing_from_snapshot": changed}}
    print(json.dumps(line), flush=True)
    ix.close()


# ---------------------------------------------------------------------------
# several batches per call, overlapped on two scratch sets
# ---------------------------------------------------------------------------

def run_pipelined(args, rounds=100):
    """The config-4 batches routed four per smetric_route_batches call on an
    index with a second scratch set, against the same batches routed one
    smetric_route_batch call each; both timed with CUDA events over `rounds`
    passes of the four batches, outputs compared bit for bit."""
    import torch
    import paper_2607_08565_gb300 as pkg
    from paper_2607_08565_gb300 import build_lib

    build_lib.build()
    torch.cuda.set_device(0)
    device = torch.device("cuda", 0)
    tr = c4_trace(args)
    p = tr.params
    host = [tr.batch(k) for k in range(N_DISTINCT_BATCHES)]
    nkeys = tr.n_prefix_blocks()
    chunk = 4096
    ix = pkg.SMetricIndex(p.num_instances, p.block_size, p.session_blocks, capacity_slots=int(nkeys / 0.7) + 1,
                          max_batch_requests=max(tr.batch_size, chunk),
                          max_batch_tokens=max(max(b.n_tokens for b in host), chunk * int(tr.prefix_len.max())),
                          hash_seed=p.hash_seed, pipeline=True)
    populate_index(ix, tr, device, chunk)
    batches = [tuple(torch.from_numpy(a).to(device) for a in (b.tokens, b.offsets, b.load)) for b in host]
    w = (p.w_load, p.w_miss, p.w_glob)
    one = [ix.route_batch(*b, w) for b in batches]
    many = ix.route_batches(batches, w)
    stream = torch.cuda.current_stream(device)

    def per_batch():
        for b, o in zip(batches, one):
            pkg.smetric_route_batch(ix.handle, b[0], b[0].numel(), b[1], b[1].numel() - 1, b[2], w,
                                    o["instance"], o["local_hit"], o["global_hit"], o["session_key"], None, 0,
                                    stream)

    def pipelined():
        ix.route_batches(batches, w, out=many, stream=stream)

    times = {}
    for name, fn in (("per_batch", per_batch), ("pipelined", pipelined)):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(rounds):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        ix.check()
        times[name] = e0.elapsed_time(e1) / (rounds * len(batches))
    for o1, o2 in zip(one, many):
        for k in o1:
            a, b = o1[k], o2[k]
            if a.dtype == torch.uint64:  # compared as int64 words (uint64 has few CUDA kernels)
                a, b = a.view(torch.int64), b.view(torch.int64)
            if not torch.equal(a, b):
                raise RuntimeError(f"smetric_route_batches differs from smetric_route_batch in {k}")
    outs = [{k: v.cpu().numpy() for k, v in o.items()} for o in one]
    algo = np.mean([algorithmic_bytes(b.lengths(), o["local_hit"], o["global_hit"], p.block_size, ix.W)["path"]
                    for b, o in zip(host, outs)])
    peak, peak_kind = peak_hbm()
    reqs = np.mean([b.n_requests for b in host])
    frac = {k: algo / (t / 1e3) / 1e9 / peak for k, t in times.items()}
    line = {"metric": METRIC, "value": reqs / (times["pipelined"] / 1e3), "unit": UNIT, "n_gpus": 1,
            "steps": rounds * len(batches), "warmup": 3 * len(batches), "ms_per_step": times["pipelined"],
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u64", "data": "synthetic",
            "per_batch_ms_per_step": times["per_batch"],
            "roofline_path": {"frac_pipelined": frac["pipelined"], "frac_per_batch": frac["per_batch"],
                              "algorithmic_bytes_per_step": float(algo), "peak": peak,
                              "peak_kind": f"{peak_kind} copy"},
            "config": {"workload": workload_name(args), "batches_per_call": len(batches),
                       "outputs_equal_per_batch_route": True}}
    print(json.dumps(line), flush=True)
    ix.close()


# ---------------------------------------------------------------------------
# session reconstruction over a config-3 trace
# ---------------------------------------------------------------------------

def run_link(args, scale=0.5):
    import torch
    import oracle
    import paper_2607_08565_gb300 as pkg
    from paper_2607_08565_gb300 import build_lib
    from synth import agent_trace
    from synth.traces import pack

    build_lib.build()
    torch.cuda.set_device(0)
    tr = agent_trace("c3_long", scale=scale, seed=7)
    p = tr.params
    reqs, users, turns = [], [], []
    for bt in tr.batches():
        for r in range(bt.n_requests):
            reqs.append(bt.tokens[bt.offsets[r]:bt.offsets[r + 1]])
        users.extend(bt.sessions.tolist())
        turns.extend(bt.turns.tolist())
    tok, off = pack(reqs)
    n = len(reqs)
    ix = pkg.SMetricIndex(p.num_instances, p.block_size, p.session_blocks, capacity_slots=1 << 16,
                          max_batch_requests=n, max_batch_tokens=len(tok), hash_seed=p.hash_seed)
    d = [torch.from_numpy(np.ascontiguousarray(a)).cuda() for a in (tok, off, np.array(users, np.int64),
                                                                    np.array(turns, np.int32))]
    for _ in range(3):
        parent, session = ix.link_sessions(*d)
    torch.cuda.synchronize()
    ix.check()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    steps = 20
    e0.record()
    for _ in range(steps):
        ix.link_sessions(*d)
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    m = min(n, 4096)  # the oracle compares every earlier request: the first two turn waves
    t0 = time.perf_counter()
    op, _ = oracle.link_sessions(p.block_size, p.hash_seed, tok[:off[m]], off[:m + 1], users[:m], turns[:m])
    dt = time.perf_counter() - t0
    if not np.array_equal(op, parent.cpu().numpy()[:m]):
        raise RuntimeError("session links differ from the oracle")
    line = {"metric": "requests linked into sessions per second (Appendix A)", "value": n / (ms / 1e3),
            "unit": "requests/s", "n_gpus": 1, "steps": steps, "warmup": 3, "ms_per_step": ms,
            "higher_is_better": True, "data": "synthetic",
            "config": {"workload": f"c3_long agent trace at scale {scale}: {n} requests, {len(tok)} tokens, "
                                   f"B = {p.block_size}, one call", "sessions": int(len(set(users))),
                       "chains": int((parent.cpu().numpy() < 0).sum())},
            "cpu_baseline": {"value": m / dt, "unit": "requests/s", "cores": 1, "kind": "oracle",
                             "sample": f"first {m} requests ({dt:.1f} s, one thread)"}}
    print(json.dumps(line), flush=True)
    ix.close()


# ---------------------------------------------------------------------------
# KV$ reuse breakdown over a whole config-2 window
# ---------------------------------------------------------------------------

def run_reuse(args, k_sessions=20):
    import torch
    import oracle
    import paper_2607_08565_gb300 as pkg
    from paper_2607_08565_gb300 import build_lib
    from synth import agent_trace
    from synth.traces import pack

    build_lib.build()
    torch.cuda.set_device(0)
    tr = agent_trace("c2_medium", scale=1.0, seed=7)
    p = tr.params
    reqs, sess = [], []
    for bt in tr.batches():
        for r in range(bt.n_requests):
            reqs.append(bt.tokens[bt.offsets[r]:bt.offsets[r + 1]])
        sess.extend(bt.sessions.tolist())
    tok, off = pack(reqs)
    n = len(off) - 1
    sys_b = np.full(n, tr.system_prompt_len // p.block_size, np.int32)
    # the oracle's sample: every turn of the first sessions, a window of its own
    keep = np.nonzero(np.asarray(sess) < k_sessions)[0]
    s_tok, s_off = pack([reqs[i] for i in keep])
    s_sess, s_sys = np.asarray(sess, np.int32)[keep], sys_b[keep]
    del reqs
    ix = pkg.SMetricIndex(p.num_instances, p.block_size, p.session_blocks, capacity_slots=1 << 16,
                          max_batch_requests=n, max_batch_tokens=len(tok), hash_seed=p.hash_seed)
    d = [torch.from_numpy(np.ascontiguousarray(a)).cuda() for a in (tok, off, np.asarray(sess, np.int32), sys_b)]
    ws = torch.empty(pkg.smetric_reuse_workspace_bytes(len(tok) // p.block_size), dtype=torch.uint8, device="cuda")
    for _ in range(3):
        out = ix.reuse_breakdown(*d, workspace=ws)
    torch.cuda.synchronize()
    ix.check()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    steps = 10
    e0.record()
    for _ in range(steps):
        ix.reuse_breakdown(*d, workspace=ws)
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    g = {k: v.cpu().numpy() for k, v in out.items()}
    if not np.array_equal(g["hit"], g["sys"] + g["intra"] + g["inter"]):
        raise RuntimeError("reuse parts do not add up")
    sg = ix.reuse_breakdown(*(torch.from_numpy(np.ascontiguousarray(a)).cuda()
                              for a in (s_tok, s_off, s_sess, s_sys)))
    ix.check()
    t0 = time.perf_counter()
    o = oracle.reuse_breakdown(p.block_size, p.hash_seed, s_tok, s_off, s_sess, s_sys)
    dt = time.perf_counter() - t0
    if any(not np.array_equal(o[k], sg[k].cpu().numpy()) for k in o):
        raise RuntimeError("reuse breakdown differs from the oracle")
    nb = int((np.diff(off) // p.block_size).sum())
    line = {"metric": "requests analysed for KV$ reuse per second (Section 3.1)", "value": n / (ms / 1e3),
            "unit": "requests/s", "n_gpus": 1, "steps": steps, "warmup": 3, "ms_per_step": ms,
            "higher_is_better": True, "data": "synthetic",
            "config": {"workload": f"c2_medium agent trace: {n} requests, {len(tok)} tokens, {nb} blocks, "
                                   f"B = {p.block_size}, one call",
                       "tokens_per_s": len(tok) / (ms / 1e3),
                       "blocks": {k: int(g[k].sum()) for k in g}},
            "cpu_baseline": {"value": len(keep) / dt, "unit": "requests/s", "cores": 1, "kind": "oracle",
                             "sample": f"every turn of sessions 0-{k_sessions - 1} ({len(keep)} requests, "
                                       f"{len(s_tok)} tokens) as a window of its own ({dt:.1f} s, one thread; "
                                       f"the oracle's cost grows with the square of the window)"}}
    print(json.dumps(line), flush=True)
    ix.close()


# ---------------------------------------------------------------------------
# windowed load imbalance over a day of running intervals
# ---------------------------------------------------------------------------

def run_imbalance(args, n_requests=3_456_000, num_instances=32, window=30_000, n_windows=2_880, sample=400_000):
    import torch
    import oracle
    import paper_2607_08565_gb300 as pkg
    from paper_2607_08565_gb300 import build_lib
    from synth import running_intervals

    build_lib.build()
    torch.cuda.set_device(0)
    inst, start, end = running_intervals(n_requests, num_instances, seed=4)
    ix = pkg.SMetricIndex(num_instances, 16, 1, capacity_slots=1 << 10, max_batch_requests=1,
                          max_batch_tokens=16)
    d = [torch.from_numpy(np.ascontiguousarray(a)).cuda() for a in (inst, start, end)]
    ws = torch.empty(pkg.smetric_imbalance_workspace_bytes(n_windows, num_instances) // 8, dtype=torch.int64,
                     device="cuda")
    for _ in range(3):
        out = ix.window_imbalance(*d, window, n_windows, workspace=ws)
    torch.cuda.synchronize()
    ix.check()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    steps = 20
    e0.record()
    for _ in range(steps):
        ix.window_imbalance(*d, window, n_windows, workspace=ws)
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    g = {k: v.cpu().numpy() for k, v in out.items()}
    # the oracle on the first requests, over the windows they reach, as a window set of its own
    m = sample
    nw_s = int(end[:m].max() // window) + 1
    t0 = time.perf_counter()
    o = oracle.window_imbalance(num_instances, window, nw_s, inst[:m], start[:m], end[:m])
    dt = time.perf_counter() - t0
    sg = ix.window_imbalance(*(x[:m] for x in d), window, nw_s)
    ix.check()
    if any(not np.array_equal(o[k], sg[k].cpu().numpy()) for k in o):
        raise RuntimeError("window imbalance differs from the oracle")
    busy = g["sum"] > 0
    imb = num_instances * g["max"][busy] / g["sum"][busy]
    line = {"metric": "requests folded into windowed load imbalance per second (Section 3.2)",
            "value": n_requests / (ms / 1e3), "unit": "requests/s", "n_gpus": 1, "steps": steps, "warmup": 3,
            "ms_per_step": ms, "higher_is_better": True, "data": "synthetic",
            "config": {"workload": f"{n_requests} running intervals over a day, {num_instances} instances, "
                                   f"{n_windows} windows of {window} ms, one call",
                       "imbalance_p50": float(np.median(imb)), "imbalance_p95": float(np.percentile(imb, 95))},
            "cpu_baseline": {"value": m / dt, "unit": "requests/s", "cores": 1, "kind": "oracle",
                             "sample": f"first {m} requests over their {nw_s} windows ({dt:.1f} s, one thread)"}}
    print(json.dumps(line), flush=True)
    ix.close()


# ---------------------------------------------------------------------------
# device-side index maintenance over a config-2 replay
# ---------------------------------------------------------------------------

def run_commit(args):
    """Route then commit on the device, batch after batch, with the capped
    tiers' evictions done by the device LRU inside the timed commit: one line
    per agent trace (c2_medium: local tiers capped, global tier uncapped;
    c3_long: both capped)."""
    import itertools
    import torch
    import paper_2607_08565_gb300 as pkg
    from paper_2607_08565_gb300 import build_lib
    from synth import agent_trace

    build_lib.build()
    torch.cuda.set_device(0)
    for name, n_batches in (("c2_medium", 24), ("c3_long", 12)):
        tr = agent_trace(name)
        p = tr.params
        batches = list(itertools.islice(tr.batches(), n_batches))
        blocks = [int((b.lengths() // p.block_size).sum()) for b in batches]
        local_cap = tr.local_cap or 0
        global_cap = tr.global_cap if (tr.global_policy == "lru" and tr.global_cap) else 0
        live = sum(blocks) if tr.global_policy == "all" or not local_cap else \
            min(sum(blocks), p.num_instances * local_cap + global_cap)
        ix = pkg.SMetricIndex(p.num_instances, p.block_size, p.session_blocks,
                              capacity_slots=max(1024, int(live / 0.6)),
                              max_batch_requests=max(b.n_requests for b in batches),
                              max_batch_tokens=max(b.n_tokens for b in batches), hash_seed=p.hash_seed)
        ix.set_lru(local_cap, global_cap)
        load = torch.zeros(p.num_instances, dtype=torch.int64, device="cuda")
        w = (p.w_load, p.w_miss, p.w_glob)
        stream = torch.cuda.current_stream()
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        route_ms, commit_ms, done = 0.0, 0.0, 0
        for k, bt in enumerate(batches):
            tok = torch.from_numpy(bt.tokens).cuda()
            off = torch.from_numpy(bt.offsets).cuda()
            torch.cuda.synchronize()
            ev[0].record(stream)
            out = ix.route_batch(tok, off, load, w, want_hashes=True)
            ev[1].record(stream)
            ix.commit_batch(off, out, also_global=tr.global_policy != "none", load=load)
            ev[2].record(stream)
            torch.cuda.synchronize()
            ix.check()
            if k >= 2:  # the first batches warm up
                route_ms += ev[0].elapsed_time(ev[1])
                commit_ms += ev[1].elapsed_time(ev[2])
                done += blocks[k]
        sizes = ix.lru_sizes().cpu().numpy()
        timed = len(batches) - 2
        line = {"metric": "device-side commit of routed batches (blocks into the chosen local tier and the "
                          "global tier, queue drain, LRU evictions of capped tiers)",
                "value": done / (commit_ms / 1e3), "unit": "blocks/s", "n_gpus": 1, "steps": timed,
                "warmup": 2, "ms_per_step": commit_ms / timed, "route_ms_per_step": route_ms / timed,
                "higher_is_better": True, "data": "synthetic",
                "config": {"workload": f"{name} agent trace ({p.num_instances} instances, B = {p.block_size}, "
                                       f"{batches[0].n_requests} requests per batch, first {n_batches} batches)",
                           "blocks_per_batch": float(np.mean(blocks[2:])), "local_cap": local_cap,
                           "global_cap": global_cap, "lru_blocks_at_end": int(sizes.sum()),
                           "evictions": "device LRU, inside the timed commit"}}
        print(json.dumps(line), flush=True)
        ix.close()


# ---------------------------------------------------------------------------
# config-5 stress sweep
# ---------------------------------------------------------------------------

SWEEP_BATCHES = (1, 4, 16, 64, 256, 1024, 4096, 8192, 16384, 32768)
SWEEP_N = (8, 16, 32, 64, 128, 256)
SWEEP_B = (16, 32, 64)


def sweep_index(N, B, table_gb, max_req, max_tok, device):
    """An index of about table_gb GB for N instances and block size B,
    holding every config-4 session prefix plus random filler keys (random
    tiers) up to load factor 0.7."""
    import torch
    import paper_2607_08565_gb300 as pkg
    from synth import burst_trace
    tr = burst_trace("c5_sweep", num_instances=N, block_size=B, batch_size=max_req)
    W = (N + 1 + 63) // 64
    entry = 16 if W == 1 else (32 if W <= 3 else 64)
    slots = int(table_gb * 1e9 / (entry + 16 / 15))  # entry + a 16-byte tag group per 15 slots
    chunk = 4096
    max_tok = max(max_tok, chunk * int(tr.prefix_len.max()))
    ix = pkg.SMetricIndex(N, B, tr.params.session_blocks, capacity_slots=slots,
                          max_batch_requests=max(max_req, chunk), max_batch_tokens=max_tok,
                          hash_seed=tr.params.hash_seed)
    populate_index(ix, tr, device, chunk)
    n_fill = int(0.7 * slots) - tr.n_prefix_blocks()
    g = torch.Generator(device=device)
    g.manual_seed(5 + N * 1000 + B)
    step = 1 << 26
    for a in range(0, max(n_fill, 0), step):
        m = min(step, n_fill - a)
        # full 64-bit range (home buckets come from a key's high bits); bit 1
        # set keeps every key >= 2
        keys = torch.randint(-(1 << 63), (1 << 63) - 1, (m,), device=device, generator=g,
                             dtype=torch.int64) | 2
        tiers = torch.randint(-1, N, (m,), device=device, generator=g, dtype=torch.int32)
        ix.insert(keys, tiers)
    ix.check()
    nb = -(-slots // 15)
    return tr, ix, nb * 15 * entry + nb * 16, tr.n_prefix_blocks() + max(n_fill, 0)


def sweep_point(tr, ix, batch, device, gpu_id=None):
    """Route one config-5 batch repeatedly; per-kernel device time, the whole
    path's roofline fraction, and the clocks sampled around the timed steps."""
    import torch
    import paper_2607_08565_gb300 as pkg
    p = tr.params
    bt = tr.batch(0, batch_size=batch)
    tok = torch.from_numpy(bt.tokens).to(device)
    off = torch.from_numpy(bt.offsets).to(device)
    load = torch.from_numpy(bt.load).to(device)
    w = (p.w_load, p.w_miss, p.w_glob)
    out = ix.route_batch(tok, off, load, w, want_hashes=False)
    ix.check()
    algo = algorithmic_bytes(bt.lengths(), out["local_hit"].cpu().numpy(), out["global_hit"].cpu().numpy(),
                             p.block_size, ix.W)
    clocks = ClockSampler(gpu_id) if gpu_id is not None else None
    if clocks:
        clocks.start()
    for _ in range(3):
        ix.route_batch(tok, off, load, w, want_hashes=False)
    ix.check()
    steps = max(5, min(200, int(2e6 / max(bt.n_tokens // p.block_size, 1))))
    stream = torch.cuda.current_stream(device)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(steps):
        ix.route_batch(tok, off, load, w, want_hashes=False)
    e1.record(stream)
    torch.cuda.synchronize()
    us = e0.elapsed_time(e1) * 1e3 / steps
    clk = None
    if clocks:
        soaked = clocks.soak(lambda i: ix.route_batch(tok, off, load, w, want_hashes=False), min_samples=4)
        clk = clocks.stop("warm-up and timed steps" + (f", then {soaked} more of the same steps (untimed)"
                                                       if soaked else ""))
    peak, peak_kind = peak_hbm()
    path_frac = algo["path"] / (us / 1e6) / 1e9 / peak
    pkg.smetric_profile_enable(ix.handle, True)
    for _ in range(steps):
        ix.route_batch(tok, off, load, w, want_hashes=False)
    prof = pkg.smetric_profile_read(ix.handle)
    pkg.smetric_profile_enable(ix.handle, False)
    ix.check()
    return {"batch": batch, "tokens": int(bt.n_tokens), "us_per_batch": us,
            "requests_per_s": batch / us * 1e6, "tokens_per_s": bt.n_tokens / us * 1e6,
            "kernels_us": {k: v[0] * 1e3 / max(v[1], 1) for k, v in prof.items()}, "steps": steps,
            "roofline_path": {"frac": path_frac, "algorithmic_bytes": algo["path"], "peak": peak,
                              "peak_kind": f"{peak_kind} copy"},
            "clocks": clk}


def run_sweep(args):
    import torch
    torch.cuda.set_device(0)
    device = torch.device("cuda", 0)
    from paper_2607_08565_gb300 import build_lib
    if not build_lib.up_to_date():
        build_lib.build()
    combos = [(64, 32, SWEEP_BATCHES)] + [(N, 32, (8192,)) for N in SWEEP_N if N != 64] + \
             [(64, B, (8192,)) for B in SWEEP_B if B != 32]
    for N, B, batches in combos:
        max_req = max(batches)
        max_tok = 0
        tr0 = None
        t0 = time.perf_counter()
        from synth import burst_trace
        tr0 = burst_trace("c5_sweep", num_instances=N, block_size=B, batch_size=max_req)
        max_tok = int(tr0.session_len.max()) * max_req
        tr, ix, table_bytes, keys = sweep_index(N, B, args.table_gb, max_req, max_tok, device)
        build_s = time.perf_counter() - t0
        try:
            gpu_id = "GPU-" + str(torch.cuda.get_device_properties(0).uuid)
        except Exception:
            gpu_id = "0"
        for b in batches:
            pt = sweep_point(tr, ix, b, device, gpu_id)
            pt.update({"sweep": "config-5", "num_instances": N, "block_size": B,
                       "table_bytes": table_bytes, "index_keys": int(keys), "build_s": build_s})
            print(json.dumps(pt), flush=True)
        ix.close()
        del ix
        torch.cuda.empty_cache()


def main():
    args = parse()
    if args.sweep:
        run_sweep(args)
        return
    if args.policy:
        run_policy(args)
        return
    if args.commit:
        run_commit(args)
        return
    if args.link:
        run_link(args)
        return
    if args.sequential:
        run_sequential(args)
        return
    if args.reuse:
        run_reuse(args)
        return
    if args.imbalance:
        run_imbalance(args)
        return
    if args.pipeline:
        run_pipelined(args)
        return
    rank, world, local, dist = dist_setup(args)
    if args.impl == "reference":
        run_reference(args, rank, world, dist)
        if dist is not None:
            dist.barrier()
            dist.destroy_process_group()
        return
    run_ours(args, rank, world, local, dist)


if __name__ == "__main__":
    main()
