"""The run-list fingerprint of include/dirigo.h, written out for the tests.

fp(list) = sum over positions k of (A * start_k + B * len_k + C) * R^k mod 2^64,
with A = 0x9E3779B97F4A7C15, B = 0xBF58476D1CE4E5B9, C = 0x94D049BB133111EB and
R = 0x2545F4914F6CDD1D.  ``fingerprints_np`` evaluates it with numpy on the
host; ``fingerprints_torch`` on the device over a whole batch, in chunks.
"""
import numpy as np

A, B, C, R = 0x9E3779B97F4A7C15, 0xBF58476D1CE4E5B9, 0x94D049BB133111EB, 0x2545F4914F6CDD1D
M64 = (1 << 64) - 1


def fp_python(runs):
    """Plain Python integers, one run list of (start, len) pairs."""
    h, rk = 0, 1
    for s, ln in runs:
        h = (h + (A * int(s) + B * int(ln) + C) * rk) & M64
        rk = (rk * R) & M64
    return h


def _powers(m):
    out = np.empty(max(m, 1), dtype=np.uint64)
    v = 1
    for k in range(max(m, 1)):
        out[k] = v
        v = (v * R) & M64
    return out


def fingerprints_np(off, runs):
    """uint64[n] for CSR offsets off[n + 1] and runs uint32[R, 2]."""
    off = np.asarray(off, dtype=np.int64)
    n = len(off) - 1
    cnt = np.diff(off)
    if len(runs) == 0:
        return np.zeros(n, dtype=np.uint64)
    k = np.arange(len(runs), dtype=np.int64) - np.repeat(off[:-1], cnt)
    w = _powers(int(cnt.max()))[k]
    with np.errstate(over="ignore"):
        t = (np.uint64(A) * runs[:, 0].astype(np.uint64) + np.uint64(B) * runs[:, 1].astype(np.uint64)
             + np.uint64(C)) * w
    out = np.zeros(n, dtype=np.uint64)
    nz = cnt > 0
    out[nz] = np.add.reduceat(t, off[:-1][nz], dtype=np.uint64)
    return out


def _signed(x):
    return x - (1 << 64) if x >= (1 << 63) else x


def fingerprints_torch(off, runs, n, chunk=1 << 26):
    """int64[n] (the uint64 bits) on the device; off int64[n + 1], runs int32 [R, 2]."""
    import torch
    dev = off.device
    total = int(off[n].item())
    cnt = off[1:n + 1] - off[:n]
    m = int(cnt.max().item()) if n else 0
    pw = torch.as_tensor(_powers(m).view(np.int64), device=dev)
    csum = torch.zeros(total + 1, dtype=torch.int64, device=dev)
    carry = torch.zeros((), dtype=torch.int64, device=dev)
    for c0 in range(0, total, chunk):
        c1 = min(total, c0 + chunk)
        idx = torch.arange(c0, c1, dtype=torch.int64, device=dev)
        loc = torch.searchsorted(off[:n + 1], idx, right=True) - 1
        k = idx - off[loc]
        r = runs[c0:c1].to(torch.int64) & 0xffffffff
        t = (r[:, 0] * _signed(A) + r[:, 1] * _signed(B) + _signed(C)) * pw[k]
        cs = torch.cumsum(t, 0) + carry
        csum[c0 + 1:c1 + 1] = cs
        carry = cs[-1].clone()
    return csum[off[1:n + 1]] - csum[off[:n]]
