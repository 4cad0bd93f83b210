"""The tests' vectorised fingerprint helpers against the definition written
with plain Python integers (the positional sum documented for d_fp in
include/dirigo.h), on random run lists, empty lists included."""
import numpy as np
import torch

from .fingerprint import fingerprints_np, fingerprints_torch, fp_python


def _lists(seed):
    rng = np.random.Generator(np.random.PCG64(seed))
    counts = rng.integers(0, 40, 300)
    counts[::17] = 0
    off = np.zeros(len(counts) + 1, dtype=np.int64)
    np.cumsum(counts, out=off[1:])
    runs = np.stack([rng.integers(0, 1 << 32, off[-1], dtype=np.uint64).astype(np.uint32),
                     rng.integers(1, 1 << 20, off[-1]).astype(np.uint32)], axis=1)
    return off, runs


def test_numpy_helper_is_the_definition():
    for seed in range(3):
        off, runs = _lists(seed)
        got = fingerprints_np(off, runs)
        want = [fp_python(runs[off[i]:off[i + 1]]) for i in range(len(off) - 1)]
        assert got.tolist() == want


def test_torch_helper_is_the_definition():
    off, runs = _lists(7)
    n = len(off) - 1
    t_off = torch.as_tensor(off)
    t_runs = torch.as_tensor(runs.view(np.int32))
    got = fingerprints_torch(t_off, t_runs, n, chunk=97).numpy().view(np.uint64)
    want = [fp_python(runs[off[i]:off[i + 1]]) for i in range(n)]
    assert got.tolist() == want
