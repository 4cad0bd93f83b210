"""Benchmark: output locations checked per second (cone + term + compare).

One step = dirigo_cone(ref) + dirigo_cone(cand) + dirigo_terms(ref) +
dirigo_terms(cand) + dirigo_compare(ref, cand, export budget) over one batch
of queried output locations, inputs resident in HBM.  The default workload is
the largest configuration: conv2d (N=128, Cin=64, 32x32, Cout=128, 3x3, pad 1)
+ bias, 2x2 max-pool, softmax over channels, every one of the 4,194,304
output locations queried; the candidate reads the weight of channels >= 96
with the wrong channel stride.  The term-key calls do not depend on the cone
calls, so by default they run on a second stream joined before the compare
(--streams 1: every call on one stream).  The per-kernel-class breakdown and
the roofline come from a second pass of the same steps on one stream with the
library's CUDA-event recording on; the headline steps run with it off.
`e2e` times the same steps with each step's queries uploaded from pinned host
memory and its verdicts and flags downloaded, the copies double-buffered on a
copy stream so that they overlap the neighbouring steps' kernels.

Multi-GPU (torchrun): the batch's slots split into contiguous ranges, one
per rank (strong scaling: the whole job checks the one batch), with no
collective on the data path; the export budget (the batch's first `budget`
undischarged slots) is split once, before timing, from every rank's
undischarged count.  Each rank still computes the term keys of every
element (the key arrays cover whole tensors), so that part of a step does
not shrink with more ranks.  The timed region is bracketed by barriers and
the slowest rank's time counts.

--impl reference times the CPU oracle on the host cores instead, on a bounded
sample of the same workload.
"""
import argparse
import json
import os
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2609_19611_gb300 import workloads as W  # noqa: E402

WORKLOAD = {
    4: "conv2d N=128 Cin=64 H=W=32 Cout=128 k=3 pad=1 + bias, maxpool 2x2, softmax over "
       "channels; candidate: weight channel stride 567 for Cout>=96; all 4,194,304 locations",
    5: "bmm B=32 M=256 K=512 N=256, sum over last dim, bias, tanh; candidate: K tiled by 64 "
       "dropping k in [480, 512); all 8,192 locations",
    3: "linear 128x1024->512, scale 0.5, LayerNorm(512); candidate: E[z^2]-mu^2 variance, "
       "split mean; 1,024 seeded locations",
    2: "conv2d N=2 Cin=3 32x32 Cout=16 + bias, GELU, sum over channels; candidate: right-edge "
       "padding off by one; 4,096 seeded locations",
    1: "X[8,16] @ W[16,8] + b, ReLU; candidate: split K, max(x,0); all 64 locations",
}
METRIC = "output locations checked/sec (cone+term+compare) and achieved HBM GB/s vs peak"
UNIT = "locations/s"


def peaks():
    """Measured copy bandwidth (GB/s) and bf16 dense rates (TFLOP/s) of this GPU
    model, else the earlier single measurement used as a fallback."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as fh:
            p = json.load(fh)
        return {"hbm_gbs": float(p["hbm_gbs"]), "bf16_tflops": float(p["bf16_tflops"]),
                "bf16_tflops_sustained": float(p["bf16_tflops_sustained"])}, "measured"
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, \
            "fallback"


# Source files whose kernels each timing class runs: a DRAM-traffic figure in
# profiles/traffic.json holds only while their digest is the one it was taken with.
CSRC = os.path.join(ROOT, "paper_2609_19611_gb300", "csrc")
CLASS_SOURCES = {
    "cone_write": ["cone.cu", "cone_prop.cuh", "cells.h", "dev.cuh", "prog.h"],
    "key_gemm": ["gemm_tc.cu", "fastdiv.h", "dev.cuh", "keyspec.cuh", "prog.h"],
    "key_limbs": ["gemm_tc.cu", "fastdiv.h", "dev.cuh", "keyspec.cuh", "prog.h"],
    "export": ["compare.cu", "cone_prop.cuh", "dev.cuh", "prog.h"],
}


def sources_digest(cls):
    import hashlib
    h = hashlib.sha256()
    for f in CLASS_SOURCES.get(cls, []):
        with open(os.path.join(CSRC, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def traffic_per_launch(cls, alg_per_launch):
    """DRAM bytes (read + write) per launch from the committed ncu capture of
    the class's kernel, scaled to this launch by its algorithmic work; None when
    there is no capture or the kernel's sources changed since."""
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as fh:
            rec = json.load(fh)[cls]
    except Exception:
        return None
    if rec.get("digest") != sources_digest(cls):
        return None
    return rec["dram_bytes"] * alg_per_launch / rec["alg_per_launch"]


class Clocks:
    """nvidia-smi sampling during the timed region."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=self.fh, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if not self.proc:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.fh.close()
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = max(mx, float(f[2]))
            except ValueError:
                continue
            for nm, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        os.unlink(self.path)
        if not sm:
            return None
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


class OracleSampler:
    """Times the oracle (both programs' cones and keys, the compare on the
    host) on random samples of configuration c's queried locations."""

    def __init__(self, c, threads):
        import oracle
        self.oracle = oracle
        ref, cand = W.config(c)
        self.R, self.C = oracle.Program(ref), oracle.Program(cand)
        self.q = W.make_queries(c, self.R.out_numel)
        self.threads = threads

    def run(self, k, seed):
        """Seconds for a sample of k locations (seeded), and its size."""
        rng = np.random.Generator(np.random.PCG64(seed))
        q, th, R, C = self.q, self.threads, self.R, self.C
        sel = q[np.sort(rng.choice(len(q), size=min(k, len(q)), replace=False))]
        t0 = time.perf_counter()
        cr, cc = R.cone_runs(sel, th), C.cone_runs(sel, th)
        kr, kc = R.keys(sel, nthreads=th), C.keys(sel, nthreads=th)
        self.oracle.compare(R, C, sel, kr, kc, cones=(cr, cc), budget=0)
        return time.perf_counter() - t0, len(sel)

    def calibrate(self, target_s, seed=0):
        """Sample size that takes about target_s seconds."""
        k = max(self.threads, 8)
        dt, m = self.run(k, seed)
        while dt < min(0.5, target_s) and m < len(self.q):
            k *= 4
            dt, m = self.run(k, seed)
        return int(min(len(self.q), max(1, m * target_s / max(dt, 1e-6))))


def oracle_rate(c, n_target_s, threads, seed=0):
    """Oracle locations/s on a bounded sample of configuration c (both
    programs: cone runs and keys; compare on the host)."""
    S = OracleSampler(c, threads)
    dt, m = S.run(S.calibrate(n_target_s, seed), seed)
    return m / dt, m, dt


def shard_queries(q, world, rank):
    """Rank `rank`'s contiguous slice of the batch q (strong scaling: the
    ranks split one batch) and its first global slot."""
    from paper_2609_19611_gb300 import shard
    lo, hi = shard.shard_range(len(q), world, rank)
    return q[lo:hi], lo


def shard_budget(n_undischarged, budget, world, rank, device=None):
    """Export budget of this rank: the batch's first `budget` undischarged
    slots are split over the ranks in slot order, which needs every rank's
    undischarged count (one all-gather of one integer per rank)."""
    import torch
    import torch.distributed as dist
    from paper_2609_19611_gb300 import shard
    if world == 1:
        return int(budget)
    mine = torch.tensor([int(n_undischarged)], dtype=torch.int64, device=device)
    every = [torch.zeros_like(mine) for _ in range(world)]
    dist.all_gather(every, mine)
    return shard.rank_budgets([int(x.item()) for x in every], int(budget))[rank]


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    threads = os.cpu_count() or 1
    per_step = []
    total = 0
    import oracle
    oracle.build()
    # one sample size for every step, so that the whole run (warm-up
    # included) takes about --ref-total-s seconds of oracle work
    step_s = max(0.05, min(args.ref_step_s, args.ref_total_s / (args.warmup + args.steps)))
    c = 4 if args.config == "all" else int(args.config)
    S = OracleSampler(c, threads)
    k = S.calibrate(step_s)
    for i in range(args.warmup + args.steps):
        dt, m = S.run(k, seed=1 + i)
        if i >= args.warmup:
            per_step.append((m, dt))
            total += m
    secs = sum(dt for _, dt in per_step)
    value = total / secs
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1000.0 * secs / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "u32", "data": "synthetic",
        "config": {"workload": WORKLOAD[c], "sample_locations_per_step":
                   total // args.steps},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                         "sample": f"{total // args.steps} random locations per step of the "
                                   f"workload, both programs' cones and keys and the compare"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default="4",
                    help="configuration 1-5, or 'all' for one line per configuration")
    ap.add_argument("--budget", type=int, default=4096)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--ref-step-s", type=float, default=6.0,
                    help="--impl reference: oracle seconds per step at most")
    ap.add_argument("--ref-total-s", type=float, default=120.0,
                    help="--impl reference: oracle seconds for the whole run")
    ap.add_argument("--streams", type=int, default=2,
                    help="1: every call on one stream; 2: term keys on a second stream")
    ap.add_argument("--graph", default="on", choices=["on", "off"],
                    help="on: each step is one replay of a CUDA graph of the batch (the "
                         "compare leaves its statistics on the device); off: the calls are "
                         "issued step by step and the compare waits for the GPU")
    ap.add_argument("--images", type=int, default=0,
                    help="config 4 only: batch of images N (default the workload's 128)")
    args = ap.parse_args()
    if args.impl == "reference":
        return run_reference(args)

    import torch
    import torch.distributed as dist
    from paper_2609_19611_gb300 import build as B
    from paper_2609_19611_gb300 import dirigo as D
    from paper_2609_19611_gb300.pipeline import BatchChecker

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    if rank == 0:
        B.build()
    if world > 1:
        dist.barrier()
    D.load()

    alu = D.alu_peak() if rank == 0 else (None, None)

    def measure(c):
        shape = {"N": args.images} if (c == 4 and args.images) else {}
        ref, cand = W.config(c, **shape)
        gr, gc = D.Graph(ref), D.Graph(cand)
        q_all = W.make_queries(c, gr.out_numel)
        n_all = len(q_all)
        workload = WORKLOAD[c] if not shape else \
            WORKLOAD[c].replace("N=128", f"N={args.images}").replace(
                "all 4,194,304", f"all {n_all:,}")
        # several ranks split the batch into contiguous slot ranges (no exchange
        # on the data path); the export budget is split once, before timing
        q, _first = shard_queries(q_all, world, rank)
        n = len(q)
        dev = torch.device("cuda", local)
        locs = torch.as_tensor(q, device=dev)
        # buffers sized once; the term keys do not depend on the cones: with
        # --streams 2 both programs' term passes run on a second stream, joined
        # before the compare; the batch waits for the GPU once, in the compare
        chk = BatchChecker(gr, gc, n, budget=0, streams=args.streams, device=dev)
        stream = chk.main
        st0 = chk.prepare(locs)   # run buffers; the undischarged count with budget 0
        chk.budget = shard_budget(st0.n_exported + st0.n_unexported, args.budget, world, rank, dev)
        chk.prepare(locs)         # the export buffer for this rank's budget
        R = [int(chk.off[i][n].item()) for i in range(2)]

        def step(overlap=True, qb=None, before_compare=None):
            qb = locs if qb is None else qb
            return chk.step(qb, overlap=overlap, before_compare=before_compare)[1]

        for _ in range(args.warmup):
            stats = step()
        torch.cuda.synchronize()
        use_graph = args.graph == "on"
        if use_graph:
            # one CUDA graph per query buffer and stream arrangement: a step is
            # one replay; its statistics are copied to pinned host memory on
            # the stream and read after the timed region
            d_locs = [locs, torch.empty_like(locs)]
            d_locs[1].copy_(locs)
            graphs = {}
            for b in (0, 1):
                for ov in ((True, False) if chk.side is not chk.main else (True,)):
                    l_cap = D.launch_count()
                    graphs[(b, ov)] = chk.capture(d_locs[b], overlap=ov)
                    if (b, ov) == (0, True):
                        # kernels of one captured step: the capture call runs the
                        # step once plainly, then records it
                        launches_per_graph = (D.launch_count() - l_cap) // 2

            def step(overlap=True, qb=None, before_compare=None, buf=0):
                graphs[(buf, overlap and chk.side is not chk.main)].replay()
                chk.read_stats(stream)
                return None

            for _ in range(args.warmup):
                step()
            torch.cuda.synchronize()
            st_, stats = chk.stats_host()
            if st_ not in (D.OK, D.E_CAPACITY) or stats.cone_error:
                D._check(st_)

        # --- device-timed region (the library's per-class event recording off)
        clocks = Clocks(local)
        l0 = D.launch_count()
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        clocks.start()
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ev0.record(stream)
        for _ in range(args.steps):
            stats = step()
        ev1.record(stream)
        torch.cuda.synchronize()
        clk = clocks.stop()
        if use_graph:
            st_, stats = chk.stats_host()
            if st_ not in (D.OK, D.E_CAPACITY) or stats.cone_error:
                D._check(st_)
        if world > 1:
            dist.barrier()
        launches = D.launch_count() - l0
        if use_graph:
            launches = launches_per_graph * args.steps   # replays issue the captured kernels
        ms = ev0.elapsed_time(ev1) / args.steps

        # --- the same steps with every call on one stream (reported beside the
        # headline when the term keys ran on a second stream)
        one_ms = None
        if chk.side is not chk.main:
            if world > 1:
                dist.barrier()
            torch.cuda.synchronize()
            ev0.record(stream)
            for _ in range(args.steps):
                step(overlap=False)
            ev1.record(stream)
            torch.cuda.synchronize()
            t1 = torch.tensor([ev0.elapsed_time(ev1) / args.steps], dtype=torch.float64, device=dev)
            if world > 1:
                dist.all_reduce(t1, op=dist.ReduceOp.MAX)
            one_ms = float(t1.item())

        # --- the same steps again on one stream with the library recording CUDA
        # events around its launches, per kernel class (the breakdown and the
        # roofline: each class's time is then its own, not shared with the other
        # stream's kernels)
        D.profile_enable(True)
        D.profile_read(reset=True)
        for _ in range(args.steps):
            chk.step(locs, overlap=False)
        torch.cuda.synchronize()
        prof = D.profile_read(reset=True)
        D.profile_enable(False)
        t = torch.tensor([ms], dtype=torch.float64, device=dev)
        if world > 1:
            dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
        if one_ms is None:
            one_ms = ms

        # --- end to end through the C ABI with host buffers (pinned).  Every step
        # copies its own queries in and its verdicts and flags out, inside the
        # timed region; the copies run on a copy stream with two query buffers, so
        # that step i+1's upload and step i's download overlap the kernels of the
        # neighbouring steps (the staging of a serving loop).  Events order every
        # reuse: an upload waits until the step that last read its buffer is
        # done, a compare until the previous step's results have been copied out.
        h_locs = torch.as_tensor(q).pin_memory()
        verdict, flags = chk.verdict[:n], chk.flags[:n]
        h_verdict = [torch.empty(n, dtype=torch.uint8).pin_memory() for _ in range(2)]
        h_flags = [torch.empty(n, dtype=torch.uint8).pin_memory() for _ in range(2)]
        if not use_graph:
            d_locs = [locs, torch.empty_like(locs)]
        cstream = torch.cuda.Stream(device=dev)
        ev_in = [torch.cuda.Event() for _ in range(2)]     # queries of a buffer uploaded
        ev_read = [torch.cuda.Event() for _ in range(2)]   # last step reading a buffer done
        ev_out = torch.cuda.Event()                        # results copied out

        def upload(i):
            with torch.cuda.stream(cstream):
                cstream.wait_event(ev_read[i & 1])
                d_locs[i & 1].copy_(h_locs, non_blocking=True)
                ev_in[i & 1].record(cstream)

        def e2e_run(k):
            upload(0)
            for i in range(k):
                stream.wait_event(ev_in[i & 1])

                def before_compare(cs, i=i):
                    if i + 1 < k:
                        upload(i + 1)
                    cs.wait_event(ev_out)

                if use_graph:
                    before_compare(stream)
                    step(buf=i & 1)
                else:
                    step(qb=d_locs[i & 1], before_compare=before_compare)
                ev_read[i & 1].record(stream)
                with torch.cuda.stream(cstream):
                    cstream.wait_event(ev_read[i & 1])
                    h_verdict[i & 1].copy_(verdict, non_blocking=True)
                    h_flags[i & 1].copy_(flags, non_blocking=True)
                    ev_out.record(cstream)

        e2e_run(2)
        torch.cuda.synchronize()
        assert torch.equal(h_verdict[1], verdict.cpu()) and torch.equal(h_flags[1], flags.cpu())
        if world > 1:
            dist.barrier()
        t0 = time.perf_counter()
        e2e_run(args.steps)
        torch.cuda.synchronize()
        e2e_ms = 1000.0 * (time.perf_counter() - t0) / args.steps
        t = torch.tensor([e2e_ms], dtype=torch.float64, device=dev)
        if world > 1:
            dist.all_reduce(t, op=dist.ReduceOp.MAX)
        e2e_ms = float(t.item())

        # --- roofline of the dominant kernel class, from the CUDA events the
        # library records around its launches on this stream over the timed steps
        pk, peak_kind = peaks()
        K = args.steps
        # per class: (bound, algorithmic work over the timed steps, launches)
        work = {
            # runs (8 B) and fingerprints (8 B) written, offsets (8 B) and
            # locations (8 B) read, per program
            "cone_write": ("hbm", K * (8.0 * (R[0] + R[1]) + 2 * 32.0 * n), 2 * K),
            # locations read, counts written
            "cone_count": ("hbm", K * 2 * 16.0 * n, 2 * K),
            # limb products over the pieces' boxes, two key lanes (one launch each)
            "key_gemm": ("tensor", K * 2 * (gr.key_tc_flops + gc.key_tc_flops),
                         2 * K * (gr.n_gemm + gc.n_gemm)),
            # limb matrices written
            "key_limbs": ("hbm", K * (gr.key_limb_bytes + gc.key_limb_bytes), None),
            # the term-list export written
            "export": ("hbm", K * float(stats.export_bytes), K),
            # SplitMix64 finalisers the key definition needs (max-sets, functions)
            "key_elem": ("alu", K * (gr.key_mix_ops + gc.key_mix_ops), None),
        }

        def roofline(cls):
            tot_ms = prof[cls][0]
            roof = {"kernel_class": cls, "ms_per_step": tot_ms / K}
            if cls not in work or tot_ms <= 0 or (work[cls][0] == "alu" and not alu[0]):
                roof.update({"bound": None, "achieved": None, "peak": None, "unit": None,
                             "frac": None, "traffic": None})
                return roof
            bound, alg, nl = work[cls]
            nl = nl or max(prof[cls][1], 1)
            if bound == "tensor":
                achieved = alg / (tot_ms * 1e-3) / 1e12
                peak, unit = pk["bf16_tflops_sustained"], "TFLOP/s"
                roof["peak_note"] = ("bf16 dense, sustained (timed inside a long step), of " +
                                     peak_kind)
            elif bound == "alu":
                achieved = alg / (tot_ms * 1e-3) / 1e9
                peak, unit = alu[0] / 1e9, "Gmix64/s"
                roof["peak_note"] = ("SplitMix64 finalisers per second, measured on this GPU "
                                     "by dirigo_alu_peak")
            else:
                achieved = alg / (tot_ms * 1e-3) / 1e9
                peak, unit = pk["hbm_gbs"], "GB/s"
                roof["peak_note"] = "copy bandwidth, of " + peak_kind
            per_launch = alg / nl
            roof.update({"bound": bound, "achieved": achieved, "peak": peak, "unit": unit,
                         "frac": achieved / peak,
                         "traffic": traffic_per_launch(cls, per_launch) if bound != "alu" else None,
                         "algorithmic_per_launch": per_launch, "launches": nl,
                         "avg_launch_ms": tot_ms / nl})
            return roof

        dom = max(prof, key=lambda k: prof[k][0])
        roof = roofline(dom)
        others = {k: roofline(k) for k in work if k != dom and prof.get(k, (0, 0))[1]}

        # whole path against the HBM bytes the method must move per batch: queries,
        # both programs' CSR offsets and runs, both root key arrays, verdicts and
        # flags, and the export
        path_bytes = (8.0 * n + 8.0 * (n + 1) * 2 + 8.0 * (R[0] + R[1]) + 8.0 * n * 2 + 2.0 * n +
                      float(stats.export_bytes))
        path_gbs = path_bytes / (ms * 1e-3) / 1e9
        hbm_path = {"bytes_per_step": path_bytes, "achieved": path_gbs, "peak": pk["hbm_gbs"],
                    "unit": "GB/s", "frac": path_gbs / pk["hbm_gbs"]}

        cpu = None
        if rank == 0 and world == 1 and not args.no_cpu_baseline:
            rate, m, dt = oracle_rate(c, args.cpu_seconds, os.cpu_count() or 1)
            cpu = {"value": rate, "unit": UNIT, "cores": os.cpu_count() or 1, "kind": "oracle",
                   "sample": f"{m} random locations of the workload ({dt:.1f} s): both programs' "
                             f"cones and keys, compare"}

        if rank == 0:
            line = {
                "metric": METRIC, "value": n_all / (ms * 1e-3), "unit": UNIT, "n_gpus": world,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
                "higher_is_better": True, "scaling": "strong", "vs_baseline": None, "dtype": "u32",
                "data": "synthetic",
                "config": {"workload": workload, "locations": n_all, "locations_rank0": n,
                           "export_budget": args.budget, "export_budget_rank0": chk.budget,
                           "export_bytes_rank0": stats.export_bytes,
                           "runs_per_step_rank0": int(R[0] + R[1]),
                           "l2": "inputs larger than L2 (run lists alone exceed 129 MB)",
                           "parallelism": f"location shards x{world} (slot ranges of one batch)",
                       "launch": ("one CUDA graph replay per step (statistics left on the device, "
                                  "copied to pinned host memory)" if use_graph else
                                  "calls issued per step; the compare waits for the GPU")},
                "roofline": roof,
                "rooflines_other": {k: {f: v[f] for f in ("ms_per_step", "bound", "achieved",
                                                          "peak", "unit", "frac", "traffic")}
                                    for k, v in others.items()},
                "alu_peak": {"mix64_per_s": alu[0], "madwide_per_s": alu[1]},
                "hbm_path": hbm_path,
                "cpu_baseline": cpu,
                "e2e": {"value": n_all / (e2e_ms * 1e-3), "unit": UNIT,
                        "h2d_bytes_per_step": 8 * n, "d2h_bytes_per_step": 2 * n},
                "one_stream": {"ms_per_step": one_ms, "value": n_all / (one_ms * 1e-3),
                               "unit": UNIT},
                "gpu_launches": int(launches),
                "clocks": clk,
                "kernels_ms_per_step": {k: v[0] / args.steps for k, v in prof.items() if v[1]},
                "verdicts": {"discharged": stats.n_discharged, "exported": stats.n_exported,
                             "unexported": stats.n_unexported},
            }
            return line
        return None

    configs = [1, 2, 3, 4, 5] if args.config == "all" else [int(args.config)]
    for c in configs:
        line = measure(c)
        if rank == 0 and line is not None:
            print(json.dumps(line), flush=True)
        torch.cuda.empty_cache()
    if world > 1:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
