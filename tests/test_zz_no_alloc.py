"""kq_assign_noalloc: the assignment step for callers that cannot allocate device
memory (for instance code running inside a host application whose allocator owns
the GPU's memory, or a service that forbids allocation once it is running), so
cannot pass a workspace. Its scratch is a fixed array built into libkq.

This file is collected last on purpose: if its GPU test fails, a run that stops
at the first failure has already run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

import synth
from paper_2003_05148_gb300 import build, kq


def test_noalloc_limits_checked_on_host():
    build.build()
    L = kq.lib()
    p = ctypes.c_void_p(1 << 20)
    assert L.kq_assign_noalloc(p, 0, p, 1, p, None, None) == 1  # n = 0
    assert L.kq_assign_noalloc(p, (1 << 24) + 1, p, 16, p, None, None) == 6  # n above the built-in scratch
    assert L.kq_assign_noalloc(p, 1 << 20, p, 65537, p, None, None) == 6  # K above the built-in scratch
    assert L.kq_assign_noalloc(ctypes.c_void_p((1 << 20) + 8), 1024, p, 16, p, None, None) == 2


@pytest.mark.gpu
def test_noalloc_matches_assign_two_calls_in_a_row():
    build.build()
    dev = torch.device("cuda:0")
    # second case takes the split-K path, so it reuses different parts of the scratch
    for n, K, seed in [(100003, 300, 1), (6000, 5000, 2)]:
        W = torch.from_numpy(synth.random_kernels(n, 9, seed, 0.1)).to(dev)
        C = torch.from_numpy(synth.random_kernels(K, 9, seed + 50, 0.1)).to(dev)
        idx_ref = torch.empty(n, dtype=torch.int32, device=dev)
        dist_ref = torch.empty(n, dtype=torch.float32, device=dev)
        ws = kq.workspace(n, K, dev)
        kq.kq_assign(W, C, idx_ref, dist_ref, ws)
        assert kq.kq_device_status(ws)[0] == 0
        idx = torch.full((n,), -1, dtype=torch.int32, device=dev)
        dist = torch.full((n,), -1.0, dtype=torch.float32, device=dev)
        kq.kq_assign_noalloc(W, C, idx, dist)
        torch.cuda.synchronize()
        # assignment parity is bit-exact in this suite: indices and distances
        assert np.array_equal(idx.cpu().numpy(), idx_ref.cpu().numpy())
        assert np.array_equal(dist.cpu().numpy().view(np.int32), dist_ref.cpu().numpy().view(np.int32))
