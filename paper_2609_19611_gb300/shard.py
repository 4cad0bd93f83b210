"""Splitting one batch of queried locations across ranks, and merging results.

Locations are checked independently (Sec. 3.4: CHECK parallelises across
locations), so a batch splits into contiguous slot ranges, one per rank, with
no exchange on the data path.  Two small host-side steps keep the merged
result equal to the one-rank result:

* the export budget is "the first E undischarged slots of the batch"; rank r
  may export only E minus the undischarged slots of ranks before it, so the
  ranks exchange their undischarged counts (one integer each) first;
* the ranks' term-list exports are merged by taking the union of their nodes
  (a node (program, tensor, element) has the same equation on every rank),
  re-sorted by (tensor, element), and concatenating the location records in
  rank order with global slot numbers.

The export byte layout ("DXP1") is documented in include/dirigo.h and read by
``parse_export``.
"""
from __future__ import annotations

import struct

__all__ = ["shard_range", "rank_budgets", "merge_stats", "parse_export", "build_export",
           "merge_exports"]

STAT_KEYS = ("n_discharged", "n_exported", "n_unexported", "n_cone_differs", "n_bot_ref",
             "n_bot_cand")


def shard_range(n, world, rank):
    """Contiguous slot range [lo, hi) of `rank` among `world` (sizes differ by <= 1)."""
    base, extra = divmod(n, world)
    lo = rank * base + min(rank, extra)
    hi = lo + base + (1 if rank < extra else 0)
    return lo, hi


def rank_budgets(undischarged_counts, budget):
    """Export budget of each rank given every rank's undischarged count."""
    out, before = [], 0
    for c in undischarged_counts:
        out.append(max(0, min(c, budget - before)))
        before += c
    return out


def merge_stats(stats):
    """Sum of per-rank stats dicts (the keys of STAT_KEYS)."""
    return {k: sum(int(s.get(k, 0)) for s in stats) for k in STAT_KEYS}


def parse_export(blob):
    """DXP1 bytes -> (programs, locations); programs[p] maps (tensor, elem) to
    (kind, fn, entries) and locations is a list of (slot, root0, root1)."""
    magic, version, total, nloc, _ = struct.unpack_from("<IIQQQ", blob, 0)
    if magic != 0x31505844 or version != 1 or total != len(blob):
        raise ValueError("not a DXP1 export")
    pos = 32
    progs = []
    for _ in range(2):
        nn, ne = struct.unpack_from("<QQ", blob, pos)
        pos += 16
        recs = []
        for _ in range(nn):
            t, kind, fn, _pad, e, b, n = struct.unpack_from("<IBBHQQQ", blob, pos)
            pos += 32
            recs.append((t, kind, fn, e, b, n))
        ents = [struct.unpack_from("<dQQ", blob, pos + 24 * i) for i in range(ne)]
        pos += 24 * ne
        nodes = {}
        for t, kind, fn, e, b, n in recs:
            nodes[(t, e)] = (kind, fn, tuple(ents[b:b + n]))
        progs.append(nodes)
    locs = [struct.unpack_from("<QQQ", blob, pos + 24 * i) for i in range(nloc)]
    return progs, locs


def build_export(progs, locs):
    """Inverse of parse_export: nodes sorted by (tensor, elem)."""
    body = b""
    for nodes in progs:
        keys = sorted(nodes)
        recs, ents = [], []
        for t, e in keys:
            kind, fn, entries = nodes[(t, e)]
            recs.append(struct.pack("<IBBHQQQ", t, kind, fn, 0, e, len(ents), len(entries)))
            ents.extend(entries)
        body += struct.pack("<QQ", len(keys), len(ents))
        body += b"".join(recs)
        body += b"".join(struct.pack("<dQQ", *x) for x in ents)
    body += b"".join(struct.pack("<QQQ", *l) for l in locs)
    total = 32 + len(body)
    return struct.pack("<IIQQQ", 0x31505844, 1, total, len(locs), 0) + body


def merge_exports(blobs, slot_offsets):
    """Merge the exports of consecutive shards (None for a rank that exported
    nothing); slot_offsets[r] is the first global slot of rank r."""
    progs = [{}, {}]
    locs = []
    for blob, off in zip(blobs, slot_offsets):
        if blob is None:
            continue
        p, l = parse_export(blob)
        for i in range(2):
            for k, v in p[i].items():
                if k in progs[i] and progs[i][k] != v:
                    raise ValueError(f"node {k} differs between shards")
                progs[i][k] = v
        locs.extend((s + off, a, b) for s, a, b in l)
    if not locs:
        return None
    return build_export(progs, locs)
