#!/usr/bin/env python
"""Benchmark of the MISA-T batched routing decision on GB300.

One step = one pass of the whole hot path over one batch: misat_route (block hash,
longest-prefix probe, caps, serial placement and admission) + misat_commit (index insert,
session update, eviction).  Workload: the throughput-stress configuration, 128
instances x 262,144 KV blocks filled to 95% (33.5M resident block hashes), batches of
65,536 mixed RLVR/RLHF/agentic requests (40/30/30), synthetic and seeded.

Every timed step starts from the same router state (a device checkpoint restored
before the step, outside the step's CUDA events), so the K steps do identical work.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl gb300|reference] [--config 1..5]

--config selects another of the five synthetic workloads (1: 4 x 2,048 blocks, 64 requests;
2: 16 x 65,536, 4,096 requests; 3: 32 x 131,072, 16,384 RLVR-heavy; 4: 64 x 262,144,
9,216 with long agentic sessions; 5, the default: the throughput stress above, whose
--n and --fill span its sweep).

Under torchrun (N > 1) every rank runs an independent replica (the path does not
shard across GPUs in this build): weak scaling, value = all ranks' requests / max time.
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
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

T_START = time.perf_counter()


def log(msg):
    print(f"[bench {time.perf_counter() - T_START:8.1f}s] {msg}", file=sys.stderr, flush=True)


METRIC = "routed requests/s (route+commit)"
UNIT = "requests/s"
CLOCK_QUERY = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
               "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
               "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")


def kernels_per_step(global_index):
    """Kernels one route+commit launches.  Route: class parameters, prologue, leaders, hash,
    caps, the block-0 probe (one kernel with the global index; with per-instance tables three:
    claim of the distinct block-0 keys, their probes, the per-request expansion), probe search,
    the four of the selection (records, initial envelopes, per-class selection, joint
    selection: it returns at once unless the per-class path hands it the batch), finalize.
    Commit: insert dedup, insert work list, insert, the global-index pass (global layout only),
    sessions, and the five eviction kernels (estimate, collect, select, delete, shift)."""
    return (12 + 9 + 1) if global_index else (14 + 9)


def max_over_ranks(ms, dist, device):
    """The largest of every rank's time (ms); the time itself on a single process.  Each rank
    runs an independent replica, so the job takes as long as its slowest rank."""
    if dist is None:
        return float(ms)
    import torch

    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank, world, steps, max_ms):
    """Units per second of the whole job: all ranks' units over the slowest rank's time."""
    return world * units_per_rank * steps / max(max_ms / 1e3, 1e-12)


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--n", type=int, default=65536, help="requests per batch")
    ap.add_argument("--fill", type=float, default=0.95, help="resident fraction of the KV block capacity")
    ap.add_argument("--e2e-steps", type=int, default=6, help="distinct batches in the end-to-end stream")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--instances", type=int, default=128, help="fewer only for small profiling captures")
    ap.add_argument("--cap", type=int, default=262144, help="blocks per instance; smaller only for profiling captures")
    ap.add_argument("--prefix-index", default="per-instance", choices=["global", "per-instance"],
                    help="block-0 probe per instance table (default: the faster step at this admission "
                         "volume) or through the global key->instance-mask index")
    ap.add_argument("--config", type=int, default=5, choices=[1, 2, 3, 4, 5],
                    help="workload: 1-4 the smaller mixed configurations, 5 the throughput stress sweep")
    return ap.parse_args()


L2_FLUSH_BYTES = 256 << 20  # twice the 129 MB L2
ROUTE_PHASES = ("prologue", "hash", "caps", "probe_first", "probe_search", "select", "finalize")
COMMIT_PHASES = ("insert", "gix_insert", "sessions", "evict")

HASH_SOURCES = ("paper_2608_11152_gb300/csrc/hash.cu", "paper_2608_11152_gb300/csrc/common.cuh")
HASH_PROFILE = os.path.join(ROOT, "profiles", "k1_block_hash_stress_n65536.md")
SELECT_SOURCES = ("paper_2608_11152_gb300/csrc/select.cu", "paper_2608_11152_gb300/csrc/envelope.cuh",
                  "paper_2608_11152_gb300/csrc/common.cuh")
SELECT_PROFILE = os.path.join(ROOT, "profiles", "k4_select_class_stress_n65536.md")


def hash_sources_sha256(files=HASH_SOURCES):
    """sha256 of a kernel's sources with comments and blank space removed (a comment edit
    does not make the committed ncu figures stale; a code edit does)."""
    import re

    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, f)) as fh:
            text = fh.read()
        text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
        text = re.sub(r"//[^\n]*", " ", text)
        h.update(" ".join(text.split()).encode())
    return h.hexdigest()


def profiled_fields(path, sources):
    """The machine-readable figures of a committed ncu summary, if that capture was taken with
    the kernel's current sources; else {}."""
    try:
        fields = {}
        for line in open(path):
            if ":" in line and line.startswith("- `"):
                k, v = line[3:].split("`:", 1)
                fields[k.strip()] = v.strip().strip("`")
        if fields.get("sources_sha256") != hash_sources_sha256(sources):
            return {}
        return fields
    except Exception:
        return {}


def profiled_hash_fields():
    """Figures of the block-hash kernel from its committed ncu summary (DRAM bytes per launch
    and the batch's token count, ALU pipe occupancy), or {}."""
    return profiled_fields(HASH_PROFILE, HASH_SOURCES)


def profiled_select_traffic(n, instances):
    """DRAM bytes per launch of the per-class selection from its committed ncu summary, when
    that capture's workload is this one (the stress batch at 128 instances), else None."""
    f = profiled_fields(SELECT_PROFILE, SELECT_SOURCES)
    if not f or int(f["batch_requests"]) != int(n) or int(f["instances"]) != int(instances):
        return None
    return int(f["traffic_bytes_per_launch"])


def profiled_traffic(batch_tokens):
    """DRAM bytes per launch of the block-hash kernel, scaled from the captured batch to this
    one by the token count (every token is read once, so the traffic grows with the tokens),
    or None without a current capture."""
    f = profiled_hash_fields()
    if "traffic_bytes_per_launch" not in f:
        return None
    return int(round(int(f["traffic_bytes_per_launch"]) * int(batch_tokens) / int(f["batch_tokens"])))


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def workload(args):
    from paper_2608_11152_gb300 import workload as wl

    if args.config == 5:
        return wl.config5(n=args.n, fill=args.fill, instances=args.instances, cap=args.cap)
    return {1: wl.config1, 2: wl.config2, 3: wl.config3, 4: wl.config4}[args.config]()


CONFIG_NAMES = {
    1: "tiny mixed batch: 4 instances x 2048 blocks, 64 requests 50/25/25",
    2: "medium mixed batch: 16 instances x 65536 blocks, 4096 requests 40/30/30",
    3: "RLVR-heavy long tail: 32 instances x 131072 blocks, 16384 requests 70/15/15, fan-out 16",
    4: "agentic-heavy long sessions: 64 instances x 262144 blocks, 1024 sessions + 8192 RLVR/RLHF, 20/20/60",
}


def workload_config(args, sc):
    if args.config == 5:
        name = (f"throughput stress: {sc.W} instances x {int(sc.cap_blocks[0])} blocks, "
                f"fill {int(round(args.fill * 100))}%, {args.n} requests/batch 40/30/30 RLVR/RLHF/agentic")
    else:
        name = CONFIG_NAMES[args.config]
    return {"workload": name,
            "instances": int(sc.W), "cap_blocks": int(sc.cap_blocks[0]), "fill": args.fill if args.config == 5 else None,
            "batch_requests": int(sc.batch.n), "batch_tokens": int(sc.batch.n_tokens), "block_tokens": 16,
            "selection": "serial in arrival order", "mode": "MISA-T", "prefix_index": args.prefix_index,
            "l2": ("L2 flushed before every timed step (a %d MB write, outside the step's events) after the "
                   "state restore; tokens %.3f GB, tables %.3f GB" % (L2_FLUSH_BYTES >> 20, sc.batch.n_tokens * 4 / 1e9,
                                                                    sc.W * 2 * int(sc.cap_blocks[0]) * 16 / 1e9))}


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 20 ms while active; the summary
    keeps the samples taken inside the timed region (mark() brackets it)."""

    def __init__(self, index):
        self.index = index
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        self.p = None
        self.t0 = self.t1 = None

    def start(self):
        try:
            self.p = subprocess.Popen(["nvidia-smi", f"--id={self.index}", f"--query-gpu={CLOCK_QUERY}",
                                       "--format=csv,noheader,nounits", "-lms", "20"], stdout=self.f,
                                      stderr=subprocess.DEVNULL)
        except Exception:
            self.p = None

    def mark(self, t0, t1):
        """Host wall-clock bounds (time.time()) of the timed region."""
        self.t0, self.t1 = t0, t1

    def stop(self):
        if self.p is not None:
            self.p.terminate()
            try:
                self.p.wait(timeout=5)
            except Exception:
                self.p.kill()
        self.f.flush()

    @staticmethod
    def parse(lines):
        """(epoch seconds, fields after the timestamp) of every well-formed sample line."""
        import datetime

        out = []
        for line in lines:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 10 or not parts[2].replace(".", "").isdigit():
                continue
            try:
                ts = datetime.datetime.strptime(parts[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
            except ValueError:
                continue
            out.append((ts, parts[1:]))
        return out

    def summary(self):
        try:
            samples = self.parse(open(self.f.name))
        except Exception:
            samples = []
        return self.summarize(samples, self.t0, self.t1)

    @staticmethod
    def summarize(samples, t0, t1):
        if not samples:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no nvidia-smi samples"], "samples": 0}
        window = "timed region"
        rows = [r for ts, r in samples if t0 is not None and t0 - 0.01 <= ts <= t1 + 0.01]
        if not rows:
            # the region was shorter than the sampling period: the samples nearest to it
            window = "nearest samples (timed region shorter than the sampling period)"
            mid = 0.5 * (t0 + t1) if t0 is not None else samples[-1][0]
            near = sorted(samples, key=lambda x: abs(x[0] - mid))[:3]
            rows = [r for _, r in near]
        sm = [float(r[1]) for r in rows]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower().startswith("active")})
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(float(r[2]) for r in rows),
                "reasons": reasons, "samples": len(rows), "window": window,
                "power_w_max": max(float(r[3]) for r in rows)}


def setup_router(sc, torch, prefix_index):
    from paper_2608_11152_gb300 import misat

    r = misat.Router(sc.cap_blocks, max_batch=sc.max_batch, max_tokens=sc.max_tokens,
                     protected_frac_q16=sc.protected_frac_q16, mode=sc.mode,
                     hold_delay_q=sc.hold_delay_q, prior_kbar=sc.prior_kbar, prior_T_us=sc.prior_T_us,
                     prefix_index=prefix_index)
    r.set_mixture(sc.rho_ppm)
    r.set_instance_state(sc.backlog_q, sc.tokcost_q, sc.contraction)
    for f in sc.fillers:
        r.load_entries(f.w, f.keys, f.metas)
    for c in sc.chains:
        r.load_chains(c.tok_off, c.tokens, c.inst, c.seq, c.arr, c.max_blocks)
    log("gpu: resident fill loaded")
    for b, c in sc.warm:
        r.route(r.device_batch(b))
        r.commit()
        r.complete(c.session, c.cls, c.total_blocks, c.residency_us, c.done)
    r.sync()
    log("gpu: warm-up batches routed and committed")
    return r


def setup_oracle(sc):
    import oracle

    o = oracle.Oracle(sc.cap_blocks, protected_frac_q16=sc.protected_frac_q16, mode=sc.mode,
                      hold_delay_q=sc.hold_delay_q, prior_kbar=sc.prior_kbar, prior_T_us=sc.prior_T_us)
    o.set_mixture(sc.rho_ppm)
    o.set_instance_state(sc.backlog_q, sc.tokcost_q, sc.contraction)
    for f in sc.fillers:
        o.load_entries(f.w, f.keys, f.metas)
    for c in sc.chains:
        o.load_chains(c.tok_off, c.tokens, c.inst, c.seq, c.arr, c.max_blocks)
    log("oracle: resident fill loaded")
    for b, c in sc.warm:
        o.route(b.cls, b.session, b.tok_off, b.tokens)
        o.commit()
        o.complete(c.session, c.cls, c.total_blocks, c.residency_us, c.done)
    log("oracle: warm-up batches routed and committed")
    return o


def cpu_step(o, b):
    t = time.perf_counter()
    o.route(b.cls, b.session, b.tok_off, b.tokens)
    o.commit()
    return time.perf_counter() - t


def algorithmic_bytes(sc, st, mask_words=None, admitted_blocks=0, evict_buckets=0, insert_ops=None):
    """Algorithmic HBM bytes per launch of the hash, probe and commit kernels (see the design
    notes).  mask_words: words per key of the global prefix index, None for the per-instance
    probe; admitted_blocks: full blocks of the admitted requests; insert_ops: the insert's key
    operations (admitted blocks less those a later request of the same instance inserts; None:
    all of them); evict_buckets: buckets of the tables above capacity after the inserts (the
    collect scan)."""
    b = sc.batch
    L = np.diff(b.tok_off)
    nb = L // 16
    n_blocks = int(nb.sum())
    # K1: every full block's 16 token ids are read once (64 B) and its key written once (8 B),
    # plus two 8-byte offsets per request
    hash_b = 72 * n_blocks + 16 * b.n
    if mask_words is None:
        # K2 phase 1 per instance: one 32-byte key group per block-0 probe of a distinct key
        # (each distinct block-0 key is probed once per instance), that key's instance mask
        # written and its slot listed; per request its H row written (2 B per pair), its
        # block-0 key, block count and key base read (the batch-local index of distinct keys
        # stays in L2 and is not counted)
        mw = (sc.W + 63) // 64
        first_b = 32 * st.probes_first + (8 * mw + 12) * st.first_block_keys + 2 * b.n * sc.W + 20 * b.n
    else:
        # K2 phase 1 through the global index: one 32-byte key group per bucket read, the mask
        # of each looked-up key, the H row, request fields (the hit list is not counted)
        first_b = 32 * st.bucket_reads_first + 8 * mask_words * st.probes_first + 2 * b.n * sc.W + 20 * b.n
    # K2 phase 2: one 32-byte key group per probe of the binary searches
    search_b = 32 * (st.probes - st.probes_first)
    mw = mask_words or 0
    ops = admitted_blocks if insert_ops is None else insert_ops
    return {
        "hash": hash_b, "probe_first": first_b, "probe_search": search_b, "n_blocks": n_blocks,
        # K3b/K4a selection: one 32-byte record per request read, the decision fields written
        "select": 32 * b.n + 10 * b.n,
        # K4b insert: per key operation, its key read (8 B), its home key group (32 B) and the
        # read-modify-write of its meta (16 B); per new key its (key, instance) entry (16 B);
        # per block left to a later request, its key and the later request's key compared (16 B)
        "insert": 56 * ops + 16 * st.new_keys + 16 * (admitted_blocks - ops),
        # global index: per new key, its entry read (16 B), a key group (32 B), its mask word RMW (16 B)
        "gix_insert": (64 * st.new_keys) if mask_words else 0,
        # K4c collect: the meta group of every bucket of a table above capacity (32 B)
        "evict_collect": 32 * evict_buckets,
        # delete: per evicted entry its key group (32 B) and slot cleared (16 B), its global-index
        # key group and mask word (32 + 8 mw B), its deleted-slot bit (8 B)
        "evict_delete": (88 + 8 * mw) * st.evicted,
        # shift: per evicted entry one bucket of its run read and written (64 + 64 B)
        "evict_shift": 128 * st.evicted,
    }


def run_gb300(args):
    import torch

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    import __graft_entry__

    if rank == 0 or world == 1:
        __graft_entry__.build()
    if dist:
        dist.barrier()
    from paper_2608_11152_gb300 import misat

    sc = workload(args)
    log(f"workload generated: {sc.name}, {sc.batch.n_tokens} tokens in the measured batch")
    # the stream of the end-to-end measurement: the measured batch, then the generator's next ones
    stream_batches = []
    if args.e2e_steps > 0 and sc.stream is not None:
        stream_batches = [(sc.batch, sc.batch_completion, sc.batch_delta)]
        while len(stream_batches) < args.e2e_steps:
            stream_batches.append(sc.stream.next_batch(sc.batch.n, delta=True))
        sc.max_tokens = max(sc.max_tokens, max(x.n_tokens for x, _, _ in stream_batches))
        log(f"stream of {len(stream_batches)} batches generated for the end-to-end measurement")
    pidx = misat.PREFIX_GLOBAL if args.prefix_index == "global" else misat.PREFIX_PER_INSTANCE
    r = setup_router(sc, torch, pidx)
    ckpt = r.checkpoint_save()
    db = r.device_batch(sc.batch)
    out = r.alloc_decisions(sc.batch.n)
    stream = r.stream
    log("checkpoint saved, batch resident")

    def step():
        r.route(db, out)
        r.commit()

    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device="cuda")

    def flush_l2():
        with torch.cuda.stream(stream):
            flush.fill_(1)

    for i in range(args.warmup):
        r.checkpoint_restore(ckpt)
        flush_l2()
        step()
    torch.cuda.synchronize()
    K = args.steps
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(K)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(K)]
    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.3)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    t_wall = time.perf_counter()
    t_epoch0 = time.time()
    for k in range(K):
        r.checkpoint_restore(ckpt)
        flush_l2()
        torch.cuda.nvtx.range_push("misat_step")
        starts[k].record(stream)
        step()
        ends[k].record(stream)
        torch.cuda.nvtx.range_pop()
        ends[k].synchronize()
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    wall = time.perf_counter() - t_wall
    sampler.mark(t_epoch0, time.time())
    time.sleep(0.05)
    sampler.stop()
    step_ms = [starts[k].elapsed_time(ends[k]) for k in range(K)]
    total_ms = float(sum(step_ms))
    log(f"timed steps done: {total_ms / K:.3f} ms/step (wall {wall:.2f} s for {K} steps incl. restores)")
    # per-phase device times (for the roofline and the phase breakdown) come from separate
    # steps with the library's phase events on: the events are kept out of the timed steps
    KP = max(1, min(K, 10))
    phase_tot = {p: 0.0 for p in misat.PHASES}
    r.set_timing(True)
    for k in range(KP):
        r.checkpoint_restore(ckpt)
        flush_l2()
        step()
        for p, v in r.phase_times().items():
            phase_tot[p] += v
    r.set_timing(False)
    r.checkpoint_restore(ckpt)
    step()  # leaves the statistics of one plain step
    torch.cuda.synchronize()
    st = r.stats()
    r.sync()
    total_ms = max_over_ranks(total_ms, dist, "cuda")
    n = sc.batch.n
    value = whole_job_rate(n, world, K, total_ms)

    # end to end through the public host API: H2D of the batch from pinned memory, route, commit,
    # D2H of the decisions, every step
    b = sc.batch
    pin = {}
    for name, arr in (("cls", b.cls), ("session", b.session.view(np.int64)), ("tok_off", b.tok_off),
                      ("tokens", b.tokens)):
        t = torch.from_numpy(arr).pin_memory()
        pin[name] = t
    from paper_2608_11152_gb300.workload import Batch

    hb = Batch(cls=pin["cls"].numpy(), session=pin["session"].numpy().view(np.uint64), group=b.group,
               tok_off=pin["tok_off"].numpy(), tokens=pin["tokens"].numpy())
    hout = {k: torch.empty(n, dtype=d).pin_memory().numpy() for k, d in
            (("inst", torch.int32), ("reason", torch.uint8), ("hit_blocks", torch.int32))}
    r.checkpoint_restore(ckpt)
    r.route_host(hb, hout)
    r.commit()
    torch.cuda.synchronize()
    # the host link itself: one plain pinned-to-device copy of the token array
    link_gbs = None
    if b.n_tokens:
        dtok = torch.empty(b.n_tokens, dtype=torch.int32, device="cuda")
        ttok = pin["tokens"]
        dtok.copy_(ttok, non_blocking=True)
        best = None
        for _ in range(3):
            l0, l1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            l0.record(stream)
            with torch.cuda.stream(stream):
                dtok.copy_(ttok, non_blocking=True)
            l1.record(stream)
            l1.synchronize()
            t = l0.elapsed_time(l1)
            best = t if best is None else min(best, t)
        link_gbs = round(b.tokens.nbytes / (best / 1e3) / 1e9, 1)
        del dtok
        log(f"host link: {link_gbs} GB/s host to device (pinned, best of 3)")
    e2e_ms = 0.0
    e2e_each = []
    for k in range(args.e2e_steps):
        r.checkpoint_restore(ckpt)
        flush_l2()
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        r.route_host(hb, hout)
        r.commit()
        e1.record(stream)
        e1.synchronize()
        e2e_ms += e0.elapsed_time(e1)
        e2e_each.append(round(e0.elapsed_time(e1), 3))
    e2e_ms = max_over_ranks(e2e_ms, dist, "cuda")
    e2e_seq = whole_job_rate(n, world, args.e2e_steps, e2e_ms)
    log(f"e2e (one call per step, copy then route) done: {e2e_ms / max(1, args.e2e_steps):.3f} ms/step {e2e_each}")

    h2d_full = int(b.cls.nbytes + b.session.nbytes + b.tok_off.nbytes + b.tokens.nbytes)
    d2h = int(n * (4 + 1 + 4))

    # end to end over a stream of distinct batches: the measured batch and the batches the
    # workload's generator produces after it, each staged from pinned host memory (the copy of
    # batch k+1 overlaps the route and commit of batch k), routed, its decisions read back to
    # host memory, committed, and followed by the completion events of its sessions; no state
    # restore anywhere, host wall clock with the device idle at both ends.  Held requests are
    # not resubmitted (the generator does not model retries).
    def pinned(a):
        return torch.from_numpy(np.ascontiguousarray(a)).pin_memory().numpy()

    def pin_batch(bb):
        return Batch(cls=pinned(bb.cls), session=pinned(bb.session.view(np.int64)).view(np.uint64), group=bb.group,
                     tok_off=pinned(bb.tok_off), tokens=pinned(bb.tokens))

    def pin_delta(dd):
        return DeltaBatch(cls=pinned(dd.cls), session=pinned(dd.session.view(np.int64)).view(np.uint64),
                          base=pinned(dd.base), delta_off=pinned(dd.delta_off), delta_tokens=pinned(dd.delta_tokens))

    def pin_comp(c):
        return Completion(session=pinned(c.session.view(np.int64)).view(np.uint64), cls=pinned(c.cls),
                          total_blocks=pinned(c.total_blocks), residency_us=pinned(c.residency_us), done=pinned(c.done))

    from paper_2608_11152_gb300.workload import Completion, DeltaBatch

    KE = len(stream_batches)
    e2e_stream = e2e_delta = stream_device = None
    stream_runs, delta_runs = [], []
    h2d_stream = h2d_delta = comp_bytes = None
    if KE > 0:
        sb = [(pin_batch(x), pin_delta(dl), pin_comp(c)) for x, c, dl in stream_batches]
        houts = [{k: torch.empty(max(1, x.n), dtype=d).pin_memory().numpy() for k, d in
                  (("inst", torch.int32), ("reason", torch.uint8), ("hit_blocks", torch.int32))} for x, _, _ in sb]
        n_stream = sum(x.n for x, _, _ in sb)
        comp_bytes = sum(int(c.session.nbytes + c.cls.nbytes + c.total_blocks.nbytes + c.residency_us.nbytes + c.done.nbytes)
                         for _, _, c in sb)
        h2d_stream = (sum(int(x.cls.nbytes + x.session.nbytes + x.tok_off.nbytes + x.tokens.nbytes) for x, _, _ in sb)
                      + comp_bytes) // KE
        h2d_delta = (sum(int(dl.cls.nbytes + dl.session.nbytes + dl.base.nbytes + dl.delta_off.nbytes +
                             dl.delta_tokens.nbytes + 8 * (dl.n + 1)) for _, dl, _ in sb) + comp_bytes) // KE

        def run_stream(delta):
            r.checkpoint_restore(ckpt)
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            stage = (lambda k, slot: r.stage_host_delta(sb[k][1], slot)) if delta else \
                    (lambda k, slot: r.stage_host(sb[k][0], slot))
            stage(0, 0)
            for k in range(KE):
                if k + 1 < KE:
                    stage(k + 1, (k + 1) % 2)
                r.route_staged(k % 2, houts[k])
                r.commit()
                c = sb[k][2]
                r.complete(c.session, c.cls, c.total_blocks, c.residency_us, c.done)
            torch.cuda.synchronize()
            return (time.perf_counter() - t0) * 1e3

        run_stream(False)  # untimed: route graphs of both slots captured
        run_stream(True)
        stream_runs = [run_stream(False) for _ in range(3)]
        delta_runs = [run_stream(True) for _ in range(3)]
        # device time of the stream's route and commit (a separate pass with phase events)
        r.set_timing(True)
        r.checkpoint_restore(ckpt)
        dev = []
        for k in range(KE):
            r.stage_host(sb[k][0], 0)
            r.route_staged(0, houts[k])
            ph = r.phase_times()
            r.commit()
            pc = r.phase_times()
            c = sb[k][2]
            r.complete(c.session, c.cls, c.total_blocks, c.residency_us, c.done)
            dev.append((sum(ph[x] for x in ROUTE_PHASES), sum(pc[x] for x in COMMIT_PHASES), ph["select"]))
        r.set_timing(False)
        stream_device = [round(sum(x[i] for x in dev) / KE, 3) for i in range(3)]
        log(f"stream device time per batch: route {stream_device[0]} ms (selection {stream_device[2]}), "
            f"commit {stream_device[1]} ms")
        sms = max_over_ranks(sorted(stream_runs)[1], dist, "cuda")
        dms = max_over_ranks(sorted(delta_runs)[1], dist, "cuda")
        e2e_stream = whole_job_rate(n_stream / KE, world, KE, sms)
        e2e_delta = whole_job_rate(n_stream / KE, world, KE, dms)
        log(f"e2e stream of {KE} batches, full layout: {[round(x / KE, 3) for x in stream_runs]} ms/batch; "
            f"delta layout: {[round(x / KE, 3) for x in delta_runs]} ms/batch")
    e2e = e2e_stream if e2e_stream is not None else e2e_seq
    h2d = h2d_stream if h2d_stream is not None else h2d_full

    # roofline: dominant kernel of the step, plus the hash and probe kernels
    peak, peak_kind = peaks()
    gidx = None
    if pidx == misat.PREFIX_GLOBAL:
        # global prefix index: size, claimed slots and the cost of one rebuild from the
        # instance tables, amortized over the steps a rebuild's headroom lasts at this
        # workload's rate of new keys (rebuilds happen outside the steady-state step)
        mw, slots, claimed = r.global_info()
        live = sum(r.index_size(w) for w in range(sc.W))
        torch.cuda.synchronize()
        g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        g0.record(stream)
        r.global_rebuild()
        g1.record(stream)
        g1.synchronize()
        rb_ms = g0.elapsed_time(g1)
        steps_between = max(1.0, (0.7 * slots - live) / max(1, st.new_keys))
        gidx = {"mask_words": mw, "slots": slots, "claimed_after_step": claimed, "live_keys": live,
                "rebuild_ms": round(rb_ms, 3), "steps_between_rebuilds": round(steps_between, 1),
                "amortized_rebuild_ms_per_step": round(rb_ms / steps_between, 4)}
        log(f"global index: {gidx}")
    # the insert's key operations: full blocks of the admitted requests; the collect's scan:
    # buckets of the tables above capacity after the inserts (the committed sizes plus the
    # evictions of the step)
    inst_h = out["inst"][: n].cpu().numpy()
    nb_all = np.diff(sc.batch.tok_off) // 16
    admitted_blocks = int(nb_all[inst_h >= 0].sum())
    evict_buckets = 0
    for w in range(sc.W):
        if r.index_size(w) >= int(sc.cap_blocks[w]):
            evict_buckets += r.table_buckets(w)
    ab = algorithmic_bytes(sc, st, mask_words=gidx["mask_words"] if gidx else None,
                           admitted_blocks=admitted_blocks, evict_buckets=evict_buckets,
                           insert_ops=int(st.insert_ops))
    phase_ms = {p: phase_tot[p] / KP for p in phase_tot}
    # one kernel per phase below (the insert phase adds the small work-list kernel)
    KERNEL_NAMES = {"hash": "k1_block_hash",
                    "probe_first": "k2_probe_first_gix" if gidx else "k2_first_claim + k2_probe_distinct + k2_probe_first_gix",
                    "probe_search": "k2_probe_search", "select": "k4_select_class", "insert": "k4_insert",
                    "gix_insert": "k4_gix_insert", "evict_collect": "k4_evict_collect",
                    "evict_delete": "k4_evict_delete", "evict_shift": "k4_evict_shift"}

    def roof(kind):
        ms = phase_ms.get(kind, 0.0)
        byts = ab.get(kind)
        if byts is None or ms <= 0:
            return None
        ach = byts / (ms / 1e3) / 1e9
        return {"bound": "hbm", "achieved": round(ach, 1), "peak": peak, "unit": "GB/s",
                "frac": round(ach / peak, 4), "traffic": None, "bytes_per_launch": int(byts),
                "ms_per_launch": round(ms, 4), "peak_kind": peak_kind, "kernel": KERNEL_NAMES[kind]}

    kernels = {k: roof(k) for k in KERNEL_NAMES}
    if kernels["hash"] is not None:
        kernels["hash"]["traffic"] = profiled_traffic(sc.batch.n_tokens)
        hf = profiled_hash_fields()
        if "alu_pipe_active_frac" in hf:
            # the kernel's actual limiter: integer ALU issue (ncu sm__pipe_alu_cycles_active)
            kernels["hash"]["alu_pipe_active_frac_ncu"] = float(hf["alu_pipe_active_frac"])
    if kernels["select"] is not None:
        if args.config == 5:
            kernels["select"]["traffic"] = profiled_select_traffic(sc.batch.n, sc.W)
        kernels["select"]["limiter"] = ("one CTA per class walks its leaders in arrival order; bound by the "
                                        "chain of headroom-exhaustion events (barrier-separated steps), not by memory")
    # dominant kernel: the largest time per launch
    dom = max((k for k in kernels if kernels[k]), key=lambda k: kernels[k]["ms_per_launch"])
    dom_roof = dict(kernels[dom])
    if dom == "hash" and dom_roof.get("traffic") is not None:
        dom_roof["traffic_source"] = "profiles/k1_block_hash_stress_n65536.md (ncu dram__bytes_read.sum + dram__bytes_write.sum)"
    if dom == "select" and dom_roof.get("traffic") is not None:
        dom_roof["traffic_source"] = "profiles/k4_select_class_stress_n65536.md (ncu dram__bytes_read.sum + dram__bytes_write.sum)"

    clocks = sampler.summary()
    line = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": round(total_ms / K, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "u64", "data": "synthetic (seeded, shaped after the paper's workloads)",
        "config": workload_config(args, sc),
        "probes_per_s": round(world * st.probes * K / (total_ms / 1e3), 1),
        "probes_definition": ("index lookups executed by the probe kernels per second: with the global "
                              "prefix index one lookup of a request's block 0 answers all instances, and "
                              "each step of a prefix search is one lookup; with per-instance tables every "
                              "(distinct block-0 key, instance) lookup counts (requests that share their "
                              "block-0 key share its lookups)"),
        "prefix_decisions_per_s": round(world * n * sc.W * K / (total_ms / 1e3), 1),
        "prefix_decisions_definition": "(request, instance) longest-cached-prefix values H computed per second",
        "e2e": {"value": round(e2e, 1), "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "api": ("misat_stage_host + misat_route_staged + misat_commit + misat_complete over a stream of "
                        f"{KE} distinct batches (the measured one and the generator's next ones), every token "
                        "copied; the copy of batch k+1 overlaps batch k; no state restore"),
                "timer": "host wall clock over the stream, device idle at both ends; median of 3 runs",
                "runs_ms_per_step": [round(x / KE, 3) for x in stream_runs] if KE > 0 else None,
                "h2d_includes": "cls, session, tok_off, tokens of each batch and the completion events that follow it",
                "delta_layout_value": round(e2e_delta, 1) if e2e_delta is not None else None,
                "delta_layout_h2d_bytes_per_step": h2d_delta,
                "delta_layout_runs_ms_per_step": [round(x / KE, 3) for x in delta_runs] if KE > 0 else None,
                "delta_layout_api": ("misat_stage_host_delta (each prompt sent as the tokens after the earlier "
                                     "prompt of the batch it extends, as the generator emits it; rebuilt on the "
                                     "GPU) + misat_route_staged + misat_commit + misat_complete, same stream"),
                "stream_device_ms_per_batch": ({"route": stream_device[0], "selection": stream_device[2],
                                                "commit": stream_device[1]} if stream_device else None),
                "sequential_value": round(e2e_seq, 1), "host_link_h2d_gbs": link_gbs,
                "sequential_h2d_bytes_per_step": h2d_full,
                "sequential_api": ("misat_route_host + misat_commit on the measured batch from the same state "
                                   "(copy, route, read-back; CUDA events)")},
        "gpu_launches": kernels_per_step(pidx == misat.PREFIX_GLOBAL) * K,
        "roofline": dom_roof,
        "kernels": kernels,
        "prefix_index": args.prefix_index,
        "global_index": gidx,
        "value_with_rebuild": (round(whole_job_rate(n, world, 1, total_ms / K + gidx["amortized_rebuild_ms_per_step"]), 1)
                               if gidx else None),
        "value_with_rebuild_definition": ("requests / (device time of route+commit + the global prefix index's "
                                          "rebuild time divided by the steps one rebuild's headroom lasts at this "
                                          "step's rate of new keys)"),
        "phase_ms": {p: round(v, 4) for p, v in phase_ms.items()},
        "clocks": clocks,
        "wall_s_timed_loop": round(wall, 3),
        "stats": {"admitted": st.n_admitted, "held": st.n_held,
                  "admitted_by_reason": dict(zip(("continuation", "new_session", "follower"),
                                                 (int(x) for x in list(st.by_reason)[:3]))),
                  "held_by_reason": dict(zip(("global_cap", "class_cap", "no_eligible", "prefer_cache",
                                              "leader_held"), (int(x) for x in list(st.by_reason)[3:8]))),
                  "admitted_by_class": dict(zip(("rlvr", "rlhf", "agentic"), (int(x) for x in st.admitted_by_class))),
                  "held_by_class": dict(zip(("rlvr", "rlhf", "agentic"), (int(x) for x in st.held_by_class))),
                  "probes": st.probes, "bucket_reads": st.bucket_reads,
                  "new_keys": st.new_keys, "evicted": st.evicted, "hit_tokens": st.hit_tokens,
                  "query_tokens": st.query_tokens, "dtv_ppm": st.dtv_ppm,
                  "admitted_blocks": admitted_blocks, "insert_key_ops": int(st.insert_ops),
                  "first_block_keys": int(st.first_block_keys),
                  "selection_path": "joint" if int(st.joint_selection) else "per-class"},
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        base = setup_oracle(sc)
        times = []
        for _ in range(3):
            o = base.clone()
            times.append(cpu_step(o, sc.batch))
            o.close()
        t = statistics.median(times)
        log(f"oracle steps: {[round(x, 2) for x in times]} s")
        line["cpu_baseline"] = {"value": round(n / t, 1), "unit": UNIT, "cores": 1, "kind": "oracle",
                                "sample": (f"median of 3 full {n}-request batches (route+commit), each from a copy "
                                           f"of the same warmed state, single-threaded C++ oracle: "
                                           f"{', '.join(f'{x:.2f}' for x in times)} s; host has {os.cpu_count()} cores"),
                                "steps_s": [round(x, 3) for x in times]}
    else:
        line["cpu_baseline"] = None
    ckpt.free()
    r.close()
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


def run_reference(args):
    """The CPU oracle, as it stands, on this host's cores: same workload, metric and unit; every
    step restarts from the same warmed state (a copy of the oracle state, untimed)."""
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if rank != 0:
        return
    sc = workload(args)
    base = setup_oracle(sc)
    # every step routes the batch's first m requests (arrival order) from the warmed state: the
    # whole batch while the run stays within about 40 full-batch steps, a proportionally
    # shorter prefix beyond that, so that any --steps/--warmup ends within a few minutes
    b = sc.batch
    m = min(b.n, max(1, (b.n * 40) // max(1, args.warmup + args.steps)))
    if m < b.n:
        from paper_2608_11152_gb300.workload import Batch

        b = Batch(cls=b.cls[:m], session=b.session[:m], group=b.group[:m], tok_off=b.tok_off[: m + 1],
                  tokens=b.tokens[: int(b.tok_off[m])])
    n = b.n
    total = 0.0
    for k in range(args.warmup + args.steps):
        o = base.clone()
        t = cpu_step(o, b)
        o.close()
        if k >= args.warmup:
            total += t
    value = n * args.steps / total
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(1e3 * total / args.steps, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u64",
        "data": "synthetic (seeded, shaped after the paper's workloads)", "config": workload_config(args, sc),
        "cpu_baseline": {"value": round(value, 1), "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": (f"each step the first {n} of the batch's {sc.batch.n} requests (route+commit) "
                                    f"from the same warmed state (single-threaded C++ oracle; host has "
                                    f"{os.cpu_count()} cores)")},
        "e2e": {"value": round(value, 1), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gb300(args)


if __name__ == "__main__":
    main()
