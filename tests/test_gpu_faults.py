"""Failure detection of the bounded device-side waits, on the GPU without a fault.

kq_test_inject_wait_fault makes a wait run out (a grid-barrier arrival that never
comes, or codeword tiles that are never streamed) with a short poll limit; the call
must return, kq_device_status must report KQ_ERR_TIMEOUT, and the same call on a
fresh workspace must give the correct result. Nothing traps or hangs: every wait
is bounded and gives up.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import bits_equal, check_indices, dev, to_dev
from paper_2003_05148_gb300 import kq

pytestmark = pytest.mark.gpu
TIMEOUT = 7


def _status(ws):
    st, flags = kq.kq_device_status(ws)
    return st, flags


def test_level_fit_grid_barrier_gives_up():
    # cooperative 6-bit quantisation: CTA 0 never arrives at a grid barrier
    K = 5000
    C = synth.random_kernels(K, 9, 81, 0.05)
    counts = synth.random_counts(K, 82, 100)
    levels = torch.empty(64, dtype=torch.float32, device=dev())
    codes = torch.empty(K, 9, dtype=torch.uint8, device=dev())
    ws = kq.workspace(K, K, dev())
    kq.kq_test_inject_wait_fault(ws, kq.TEST_SKIP_ARRIVAL, 2000)
    kq.kq_quantize_codebook_6bit(to_dev(C), to_dev(counts), 100, levels, codes, None, ws)
    st, flags = _status(ws)
    assert st == TIMEOUT and flags & kq.FLAG_TIMEOUT
    # the same call on a fresh workspace is correct
    ws2 = kq.workspace(K, K, dev())
    kq.kq_quantize_codebook_6bit(to_dev(C), to_dev(counts), 100, levels, codes, None, ws2)
    assert _status(ws2)[0] == 0
    lv_ref, cd_ref, _ = oracle.level_fit(C, counts)
    assert bits_equal(levels.cpu().numpy(), lv_ref)
    assert np.array_equal(codes.cpu().numpy(), cd_ref)


def test_small_fit_grid_barrier_gives_up():
    # one-launch fit of the 64x64 layer (K = 16): its grid barriers run out
    lay = synth.workload(1).layers[0]
    W, sel = synth.layer_inputs(lay)
    C0 = oracle.gather_rows(W, sel)
    n, K, T = lay.n, lay.K, 3
    C = torch.empty(K, 9, dtype=torch.float32, device=dev())
    idx = torch.empty(n, dtype=torch.int32, device=dev())
    counts = torch.empty(K, dtype=torch.int32, device=dev())
    ws = kq.workspace(n, K, dev())
    kq.kq_test_inject_wait_fault(ws, kq.TEST_SKIP_ARRIVAL, 2000)
    kq.kq_fit_codebook(to_dev(W), to_dev(C0), T, C, idx, counts, None, ws)
    st, flags = _status(ws)
    assert st == TIMEOUT and flags & kq.FLAG_TIMEOUT
    ws2 = kq.workspace(n, K, dev())
    kq.kq_fit_codebook(to_dev(W), to_dev(C0), T, C, idx, counts, None, ws2)
    assert _status(ws2)[0] == 0
    C_ref, _, _, _ = oracle.fit(W, C0, T)
    scale = np.maximum(np.abs(C_ref).max(axis=1, keepdims=True), 1e-30)
    assert np.all(np.abs(C.cpu().numpy() - C_ref) <= 1e-5 * scale)


@pytest.mark.parametrize("case", ["assign", "pruned_fit"])
def test_tensor_core_assign_tile_wait_gives_up(case):
    # the codeword tiles after the first ones never arrive: the MMA issuers' waits run
    # out, every role drains, TMEM is freed, the call returns
    n, K = (65536, 2048) if case == "assign" else (40000, 4096)
    lay = synth.Layer("f", 64, n // 64, K, 4 * K, 90)
    W = synth.conv_weights(lay)
    C0 = oracle.gather_rows(W, synth.init_selection(n, K, 91))
    Wd, Cd = to_dev(W), to_dev(C0)
    idx = torch.empty(n, dtype=torch.int32, device=dev())
    dist = torch.empty(n, dtype=torch.float32, device=dev())
    C = torch.empty_like(Cd)
    counts = torch.empty(K, dtype=torch.int32, device=dev())

    def run(ws):
        if case == "assign":
            kq.kq_assign(Wd, Cd, idx, dist, ws)
        else:
            kq.kq_fit_codebook(Wd, Cd, 2, C, idx, counts, None, ws, flags=kq.FIT_PRUNE)

    ws = kq.workspace(n, K, dev())
    kq.kq_test_inject_wait_fault(ws, kq.TEST_STOP_TILE_STREAM, 20000)
    run(ws)
    st, flags = _status(ws)
    assert st == TIMEOUT and flags & kq.FLAG_TIMEOUT
    ws2 = kq.workspace(n, K, dev())
    run(ws2)
    assert _status(ws2)[0] == 0
    if case == "assign":
        rows = np.sort(synth.below(synth.stream_key(90, 3), 4096, n))
        idx_ref, dist_ref = oracle.assign(W[rows], C0, threads=oracle.default_threads())
        assert check_indices(W, C0, idx.cpu().numpy()[rows], idx_ref, rows) == 0
    else:
        ws3 = kq.workspace(n, K, dev())
        C3 = torch.empty_like(Cd)
        idx3 = torch.empty_like(idx)
        kq.kq_fit_codebook(Wd, Cd, 2, C3, idx3, counts, None, ws3)
        assert _status(ws3)[0] == 0
        assert torch.equal(C, C3) and torch.equal(idx, idx3)


def test_inject_arguments():
    ws = kq.workspace(1024, 16, dev())
    with pytest.raises(kq.KQError):
        kq.kq_test_inject_wait_fault(ws, 0x4, 100)
    kq.kq_test_inject_wait_fault(ws, 0, 0)  # clearing is always allowed
    assert _status(ws)[0] == 0
