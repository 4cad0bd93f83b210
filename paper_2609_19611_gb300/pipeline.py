"""One batch of queried locations through the whole check on one GPU.

A step is the per-location check of Sec. 3.4 for every location of a batch:
both programs' cones (``dirigo_cone_async``, one status word for the two),
both programs' term keys (``dirigo_terms``), then ``dirigo_compare`` with the
cones, their status word and the export of the first ``budget`` undischarged
locations.  The batch waits for the GPU once, inside the compare.  The term
keys do not depend on the cones, and the verdicts and the export need only
the keys: with two streams the key passes and the compare run on a second
stream, forked from the caller's stream; the cones run on the caller's
stream and an event recorded after them is handed to the compare, whose
flag passes (the only part that reads the cones) wait for it.  The second
stream is joined back into the caller's before the step returns.

Buffers are allocated once.  The run buffers are sized from the graphs'
``max_runs_per_location`` when every cone cell has a fast plan, otherwise
by a counting ``dirigo_cone`` call on the first batch; a later batch whose
runs do not fit (the compare reports the cones' ``DIRIGO_CONE_ERR_RUNS``)
grows them from the totals the prefix sum left on the device and is run
again.  The export buffer is sized by a first compare without one.

Only marshalling and stream arrangement live here; every step of the check
runs in the CUDA library.
"""
from __future__ import annotations

import ctypes

import torch

from . import dirigo as D



class BatchChecker:
    """Buffers and streams for batches of ``n`` locations of a program pair."""

    def __init__(self, gr, gc, n, budget=4096, streams=2, device=None):
        self.gr, self.gc, self.n, self.budget = gr, gc, int(n), int(budget)
        dev = torch.device(device) if device is not None else torch.device(
            "cuda", torch.cuda.current_device())
        self.dev = dev
        n = self.n
        self.ws_cone = torch.empty(max(gr.workspace_size(D.CALL_CONE, n),
                                       gc.workspace_size(D.CALL_CONE, n), 1),
                                   dtype=torch.uint8, device=dev)
        self.ws_terms = [torch.empty(max(g.workspace_size(D.CALL_TERMS, n), 1),
                                     dtype=torch.uint8, device=dev) for g in (gr, gc)]
        self.ws_cmp = torch.empty(max(D.compare_workspace_size(gr, gc, n), 1), dtype=torch.uint8,
                                  device=dev)
        self.off = [torch.empty(n + 1, dtype=torch.int64, device=dev) for _ in range(2)]
        self.fp = [torch.empty(max(n, 1), dtype=torch.int64, device=dev) for _ in range(2)]
        self.keys = [torch.empty((max(n, 1), 2), dtype=torch.int32, device=dev)
                     for _ in range(2)]
        self.verdict = torch.empty(max(n, 1), dtype=torch.uint8, device=dev)
        self.flags = torch.empty(max(n, 1), dtype=torch.uint8, device=dev)
        self.status = torch.zeros(1, dtype=torch.int32, device=dev)
        self.cap = [0, 0]
        self.runs = [None, None]
        self.exp_cap = 0
        self.exp_buf = None
        self.main = torch.cuda.current_stream(dev)
        self.side = torch.cuda.Stream(device=dev) if streams > 1 else self.main
        for i, g in enumerate((gr, gc)):
            if g.max_runs_per_location > 0:
                self._alloc_runs(i, n * g.max_runs_per_location)

    # ------------------------------------------------------------ buffers
    def _alloc_runs(self, i, cap):
        self.cap[i] = int(cap)
        self.runs[i] = torch.empty(max(self.cap[i], 1) * 2, dtype=torch.int32, device=self.dev)

    def count_runs(self, locs):
        """Run totals of both programs for this batch (a counting dirigo_cone
        call each; it waits for the stream)."""
        P = D._ptr
        out = []
        for i, g in enumerate((self.gr, self.gc)):
            st, tot = D.dirigo_cone(g, P(locs), self.n, P(self.off[i]), None, 0, None,
                                    P(self.ws_cone), self.ws_cone.numel(), D._stream(self.main))
            if st not in (D.OK, D.E_CAPACITY):
                D._check(st)
            out.append(int(tot))
        return out

    def prepare(self, locs):
        """Size every buffer for this batch (run buffers where the graphs give
        no bound, then the export by a compare without an export buffer)."""
        if self.runs[0] is None or self.runs[1] is None:
            tot = self.count_runs(locs)
            for i in range(2):
                if self.runs[i] is None or self.cap[i] < tot[i]:
                    self._alloc_runs(i, tot[i])
        st, stats = self.step(locs, export_capacity=0)
        self.exp_cap = int(stats.export_required)
        self.exp_buf = torch.empty(max(self.exp_cap, 1), dtype=torch.uint8, device=self.dev) \
            if self.exp_cap else None
        return stats

    # ------------------------------------------------------------ one step
    def enqueue_cones(self, locs, stream):
        P, s = D._ptr, D._stream(stream)
        for i, g in enumerate((self.gr, self.gc)):
            D._check(D.dirigo_cone_async(g, P(locs), self.n, P(self.off[i]), P(self.runs[i]),
                                         self.cap[i], P(self.fp[i]), P(self.status),
                                         P(self.ws_cone), self.ws_cone.numel(), s))

    def enqueue_terms(self, locs, stream):
        P, s = D._ptr, D._stream(stream)
        for i, g in enumerate((self.gr, self.gc)):
            D._check(D.dirigo_terms(g, P(locs), self.n, P(self.keys[i]), P(self.ws_terms[i]),
                                    self.ws_terms[i].numel(), s))

    def compare(self, locs, export_capacity, stream, cones_ready=None):
        P = D._ptr
        ev = ctypes.c_void_p(cones_ready.cuda_event) if cones_ready is not None else None
        return D.dirigo_compare(self.gr, self.gc, P(locs), self.n, P(self.keys[0]),
                                P(self.keys[1]),
                                (P(self.off[0]), P(self.runs[0]), P(self.fp[0])),
                                (P(self.off[1]), P(self.runs[1]), P(self.fp[1])),
                                P(self.verdict), P(self.flags), self.budget,
                                P(self.exp_buf) if export_capacity else None, export_capacity,
                                P(self.ws_cmp), self.ws_cmp.numel(), D._stream(stream),
                                d_cone_status=P(self.status), cones_ready=ev)

    def step(self, locs, export_capacity=None, overlap=True, before_compare=None):
        """One batch: (status, stats).  The status is OK, or E_CAPACITY when
        the export did not fit; any other error raises.  before_compare(s), if
        given, is called with the stream the compare is enqueued on, just
        before it is."""
        if export_capacity is None:
            export_capacity = self.exp_cap
        for _ in range(2):
            main = self.main
            side = self.side if overlap else main
            self.status.zero_()
            ready = None
            if side is not main:
                side.wait_stream(main)
            self.enqueue_terms(locs, side)
            self.enqueue_cones(locs, main)
            if side is not main:
                ready = torch.cuda.Event()
                ready.record(main)
            if before_compare is not None:
                before_compare(side)
            st, stats = self.compare(locs, export_capacity, side, ready)
            if side is not main:
                main.wait_stream(side)
            if stats.cone_error == D.CONE_ERR_RUNS:
                # the runs did not fit: grow from the totals left on the device
                for i in range(2):
                    tot = int(self.off[i][self.n].item())
                    if tot > self.cap[i]:
                        self._alloc_runs(i, tot)
                continue
            if stats.cone_error or st not in (D.OK, D.E_CAPACITY):
                D._check(st)
            return st, stats
        raise D.DirigoError(D.E_CAPACITY, "cone runs still do not fit after resizing")

    # ------------------------------------------------------------ graphs
    def enqueue_step(self, locs, main, export_capacity=None, overlap=True):
        """One batch enqueued on `main` with no host wait: the compare is
        dirigo_compare_async, whose statistics and status land in device
        memory (self.dstats, self.dstatus)."""
        if export_capacity is None:
            export_capacity = self.exp_cap
        side = self.side if overlap else main
        self.status.zero_()
        ready = None
        if side is not main:
            side.wait_stream(main)
        self.enqueue_terms(locs, side)
        self.enqueue_cones(locs, main)
        if side is not main:
            ready = torch.cuda.Event()
            ready.record(main)
        P = D._ptr
        ev = ctypes.c_void_p(ready.cuda_event) if ready is not None else None
        D._check(D.dirigo_compare_async(
            self.gr, self.gc, P(locs), self.n, P(self.keys[0]), P(self.keys[1]),
            (P(self.off[0]), P(self.runs[0]), P(self.fp[0])),
            (P(self.off[1]), P(self.runs[1]), P(self.fp[1])), P(self.verdict), P(self.flags),
            self.budget, P(self.exp_buf) if export_capacity else None, export_capacity,
            P(self.dstats), P(self.dstatus), P(self.ws_cmp), self.ws_cmp.numel(),
            D._stream(side), d_cone_status=P(self.status), cones_ready=ev))
        if side is not main:
            main.wait_stream(side)

    def capture(self, locs, overlap=True):
        """A CUDA graph of one batch over the fixed buffer `locs` (sized by
        prepare() first).  Replaying it runs every kernel of the batch with one
        launch from the host; the statistics stay on the device."""
        if not hasattr(self, "dstats"):
            self.dstats = torch.zeros(9, dtype=torch.int64, device=self.dev)
            self.dstatus = torch.zeros(1, dtype=torch.int32, device=self.dev)
            self.hstats = torch.zeros(10, dtype=torch.int64).pin_memory()
        # the library's internal streams and attributes are set up on a plain
        # run before capture
        self.enqueue_step(locs, self.main, overlap=overlap)
        torch.cuda.synchronize(self.dev)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.enqueue_step(locs, torch.cuda.current_stream(self.dev), overlap=overlap)
        torch.cuda.synchronize(self.dev)
        return g

    def read_stats(self, stream=None):
        """Copy the device statistics of the last batch into pinned host memory
        on `stream` (no wait); stats_host() reads them after a synchronize."""
        s = stream or torch.cuda.current_stream(self.dev)
        with torch.cuda.stream(s):
            self.hstats[:9].copy_(self.dstats, non_blocking=True)
            self.hstats[9:10].copy_(self.dstatus.to(torch.int64), non_blocking=True)

    def stats_host(self):
        """(status, CompareStats) from the last read_stats() copy."""
        v = self.hstats.tolist()
        st = D.CompareStats(*v[:9])
        return int(v[9]), st

    # ------------------------------------------------------------ results
    def cones(self, i, total=None):
        """(offsets, runs [R, 2] int32 view, fingerprints) of program i."""
        tot = int(self.off[i][self.n].item()) if total is None else total
        return self.off[i], self.runs[i][:2 * tot].view(tot, 2), self.fp[i][:self.n]

    def blob(self, stats):
        if self.exp_buf is None or not stats.export_bytes:
            return None
        return self.exp_buf[:stats.export_bytes]
