"""The C ABI without a GPU: the library loads, exports what include/kq.h declares,
validates arguments on the host, and its storage report matches the oracle and
the paper's tables."""
import ctypes
import os
import re
from fractions import Fraction

import numpy as np
import pytest

import oracle
import synth
from paper_2003_05148_gb300 import build, kq

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "kq.h")


@pytest.fixture(scope="module")
def lib():
    build.build()
    return kq.lib()


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(kq_[a-z0-9_]+)\s*\(", text)))


def test_exports_every_declared_symbol(lib):
    names = _declared()
    assert len(names) >= 12
    for name in names:
        assert hasattr(lib, name), name
    assert sorted(kq.EXPORTS) == names


def test_status_strings_and_version(lib):
    assert kq.kq_abi_version() == 7
    for code, name in kq.STATUS_NAMES.items():
        assert kq.kq_status_string(code) == name
    assert kq.kq_status_string(99) == "KQ_ERR_UNKNOWN"


def test_workspace_bytes_rules(lib):
    assert kq.kq_workspace_bytes(0, 1) == 0
    assert kq.kq_workspace_bytes(10, 11) == 0  # K > n
    assert kq.kq_workspace_bytes(10, 0) == 0
    assert kq.kq_workspace_bytes(2 ** 31, 16) == 0
    a = kq.kq_workspace_bytes(4096, 16)
    b = kq.kq_workspace_bytes(4194304, 65536)
    assert 4096 < a < b and a % 256 == 0 and b % 256 == 0


@pytest.mark.parametrize("n,K,seed", [(1, 1, 0), (50, 50, 9), (4096, 16, 1001), (65536, 256, 1202),
                                     (4194304, 65536, 1502), (2 ** 31 - 1, 300, 2 ** 64 - 1), (10, 3, 12345)])
def test_seed_indices_match_the_input_generator(lib, n, K, seed):
    # the library's draw and the seeded input module's are written separately from
    # the same definition (SplitMix64 stream 4, partial Fisher-Yates)
    got = kq.kq_seed_indices(n, K, seed).numpy()
    assert np.array_equal(got, synth.init_selection(n, K, seed))
    assert len(np.unique(got)) == K and got.min() >= 0 and got.max() < n


def test_seed_indices_rejects_bad_sizes(lib):
    out = (ctypes.c_int64 * 4)()
    assert lib.kq_seed_indices(0, 1, 1, out) == 1
    assert lib.kq_seed_indices(3, 4, 1, out) == 1
    assert lib.kq_seed_indices(2 ** 31, 1, 1, out) == 1
    assert lib.kq_seed_indices(10, 0, 1, out) == 1
    assert lib.kq_seed_indices(10, 2, 1, None) == 1


def test_host_validation_before_any_device_work(lib):
    # Bad arguments are rejected on the host; the fake pointers are never touched.
    L = lib
    good = ctypes.c_void_p(1 << 20)  # 256-byte aligned dummy address
    odd = ctypes.c_void_p((1 << 20) + 4)
    ws_bytes = kq.kq_workspace_bytes(1024, 16)
    assert L.kq_assign(good, 0, good, 16, None, good, None, good, ws_bytes, None) == 1  # n = 0
    assert L.kq_assign(good, 1024, good, 2048, None, good, None, good, ws_bytes, None) == 1  # K > n
    assert L.kq_assign(odd, 1024, good, 16, None, good, None, good, ws_bytes, None) == 2  # W not 16-byte aligned
    assert L.kq_assign(good, 1024, good, 16, ctypes.c_void_p((1 << 20) + 2), good, None, good, ws_bytes, None) == 2
    assert L.kq_assign(good, 1024, good, 16, None, good, None, None, ws_bytes, None) == 6  # no workspace
    assert L.kq_assign(good, 1024, good, 16, None, good, None, good, ws_bytes - 1, None) == 6  # too small
    assert L.kq_assign(good, 1024, good, 16, None, good, None, odd, ws_bytes, None) == 2  # ws alignment
    assert L.kq_update_centroids(good, 1024, good, 16, None, good, good, good, ws_bytes, None) == 1
    assert L.kq_fit_codebook(good, 1024, 16, good, -1, 0, good, good, good, None, None, good, ws_bytes, None) == 1
    assert L.kq_fit_codebook(good, 1024, 16, good, 3, 7, good, good, good, None, None, good, ws_bytes, None) == 1
    assert L.kq_fit_codebook(good, 1024, 16, good, 3, 4, good, good, good, None, None, good, ws_bytes, None) == 1
    assert L.kq_quantize_codebook_6bit(good, 16, good, -1, good, good, None, good, ws_bytes, None) == 1
    assert L.kq_quantize_codebook_6bit(good, 16, good, 10, good, good, None, good, 100, None) == 6
    assert L.kq_reconstruct(good, 1024, None, 16, None, None, good, good, ws_bytes, None) == 1  # nothing to decode
    assert L.kq_reconstruct(good, 1024, good, 16, good, None, good, good, ws_bytes, None) == 1  # codes w/o levels
    assert L.kq_reconstruct(good, 1024, good, 16, None, None, odd, good, ws_bytes, None) == 2  # W_out alignment
    assert L.kq_init_codebook(good, 1024, good, 2000, good, good, ws_bytes, None) == 1
    assert L.kq_device_status(None, 0, None, None) == 6
    u64 = ctypes.c_uint64()
    assert L.kq_fit_prune_stats(None, 0, ctypes.byref(u64), ctypes.byref(u64), None) == 6  # no workspace
    assert L.kq_fit_prune_stats(good, 4096, None, ctypes.byref(u64), None) == 1  # no output
    assert L.kq_fit_prune_stats(odd, 4096, ctypes.byref(u64), ctypes.byref(u64), None) == 2  # ws alignment
    assert L.kq_fit_prune_stats(good, 4095, ctypes.byref(u64), ctypes.byref(u64), None) == 6  # too small
    nan = float("nan")
    assert L.kq_quantize_scalars_6bit(good, 0, 10, good, good, None, good, 4096, None) == 1  # m = 0
    assert L.kq_quantize_scalars_6bit(good, 100, 100001, good, good, None, good, 4096, None) == 1
    assert L.kq_quantize_scalars_6bit(good, 100, 10, good, good, None, good, 4095, None) == 6
    assert L.kq_codebook_grad_step(good, 1024, good, 16, nan, good, good, good, good, ws_bytes, None) == 1  # lr NaN
    assert L.kq_codebook_grad_step(good, 1024, good, 16, float("inf"), good, good, good, good, ws_bytes, None) == 1
    assert L.kq_codebook_grad_step(odd, 1024, good, 16, 0.1, good, good, good, good, ws_bytes, None) == 2
    assert L.kq_codebook_grad_step(good, 1024, good, 16, 0.1, good, good, good, good, ws_bytes - 1, None) == 6
    assert L.kq_levels_grad_step(good, 0, good, 16, good, 0.1, good, good, None, good, 4096, None) == 1
    assert L.kq_levels_grad_step(good, 1024, good, 16, None, 0.1, good, good, None, good, 4096, None) == 1
    assert L.kq_levels_grad_step(good, 1024, good, 16, good, nan, good, good, None, good, 4096, None) == 1
    assert L.kq_levels_grad_step(odd, 1024, good, 16, good, 0.1, good, good, None, good, 4096, None) == 2
    assert L.kq_levels_grad_step(good, 1024, good, 16, good, 0.1, good, good, ctypes.c_void_p((1 << 20) + 4),
                                 good, 4096, None) == 2  # counts not 8-byte aligned
    assert L.kq_levels_grad_step(good, 1024, good, 16, good, 0.1, good, good, None, good, 4095, None) == 6
    QR = L.kq_quantize_reconstruct
    assert QR(good, 1024, good, 16, None, None, good, good, ws_bytes, None) == 1  # no levels
    assert QR(good, 1024, good, 2048, good, None, good, good, ws_bytes, None) == 1  # K > n
    assert QR(good, 1024, good, 16, good, None, odd, good, ws_bytes, None) == 2  # W_out alignment
    assert QR(good, 1024, good, 16, good, None, good, good, ws_bytes - 1, None) == 6
    ws_s = kq.kq_workspace_bytes(1024, 256)
    S = L.kq_search_codebook_size
    assert S(good, 1024, good, 256, 0.0, 0.5, 8, 3, good, good, good, ctypes.byref(ctypes.c_int32()), None, None, None,
             None, good, ws_s, None) == 1  # alpha = 0
    assert S(good, 1024, good, 256, 0.25, -0.5, 8, 3, good, good, good, ctypes.byref(ctypes.c_int32()), None, None,
             None, None, good, ws_s, None) == 1  # r < 0
    assert S(good, 1024, good, 256, 0.25, 0.5, 65, 3, good, good, good, ctypes.byref(ctypes.c_int32()), None, None,
             None, None, good, ws_s, None) == 1  # too many steps
    assert S(good, 1024, good, 255, 0.25, 0.5, 8, 3, good, good, good, ctypes.byref(ctypes.c_int32()), None, None,
             None, None, good, ws_s, None) == 1  # sel shorter than N_init = 256
    assert S(good, 1024, good, 256, 0.25, 0.5, 8, 3, good, good, good, None, None, None, None, None, good, ws_s,
             None) == 1  # no K output
    assert S(odd, 1024, good, 256, 0.25, 0.5, 8, 3, good, good, good, ctypes.byref(ctypes.c_int32()), None, None,
             None, None, good, ws_s, None) == 2
    assert S(good, 1024, good, 256, 0.25, 0.5, 8, 3, good, good, good, ctypes.byref(ctypes.c_int32()), None, None,
             None, None, good, ws_s - 1, None) == 6


def _report_rows():
    rows = []
    with open(os.path.join(os.path.dirname(__file__), "golden", "paper_tables.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                p = line.split()
                rows.append((int(p[2]), int(p[3])))
    return rows


@pytest.mark.parametrize("n,k", _report_rows() + [(1, 1), (7, 3), (2 ** 30, 2), (4194304, 65536), (4096, 4096)])
@pytest.mark.parametrize("b_c", [32, 6])
def test_report_matches_oracle(lib, n, k, b_c):
    got = kq.kq_compression_report(n, k, 3, b_c)
    ref = oracle.report(n, k, 3, b_c)
    assert got["index_bits"] == ref.index_bits
    assert got["codebook_bits"] == ref.codebook_bits
    assert got["total_bits"] == ref.total_bits
    assert Fraction(got["beta"]) == pytest.approx(ref.beta, rel=1e-15)
    assert Fraction(got["ratio_kq"]) == pytest.approx(ref.ratio_kq, rel=1e-15)
    # Eq. 5 at its limit (u = 2 fp32 entries, one bit per weight) for the same layer
    assert Fraction(got["ratio_con_1bit"]) == pytest.approx(oracle.ratio_conventional(n, 3, 2, 32), rel=1e-15)


def test_conventional_ratio_matches_oracle(lib):
    for n, u, b1 in [(4096, 2, 32), (10 ** 9, 2, 32), (65536, 4, 32), (192, 16, 6)]:
        assert kq.kq_conventional_ratio(n, 3, u, b1) == pytest.approx(float(oracle.ratio_conventional(n, 3, u, b1)),
                                                                      rel=1e-15)
    with pytest.raises(kq.KQError):
        kq.kq_conventional_ratio(10, 3, 1, 32)
    with pytest.raises(kq.KQError):
        kq.kq_compression_report(0, 4)


def _job(base, **kw):
    g = lambda a: ctypes.c_void_p((1 << 20) + (base << 12) + a)  # distinct 256-byte aligned dummies
    d = dict(W=g(0), n=1024, K=16, sel=None, C=g(256), idx=g(512), counts=g(768), objective=None, levels=None,
             codes=None, W_out=None, ws=g(1024), ws_bytes=kq.kq_workspace_bytes(1024, 16))
    d.update(kw)
    return kq.LayerJob(**d)


def test_fit_layers_arguments_checked_on_host(lib):
    # every rejection happens before any CUDA call (the dummy pointers are never used)
    assert ctypes.sizeof(kq.LayerJob) == 104  # the C struct: 12 pointer-sized fields and n, K (padded)
    FL = lib.kq_fit_layers
    one = (kq.LayerJob * 1)(_job(1))
    assert FL(None, 1, 3, 10, 0, None) == 1
    assert FL(one, 0, 3, 10, 0, None) == 1
    assert FL(one, 1, -1, 10, 0, None) == 1
    assert FL(one, 1, 3, 100001, 0, None) == 1
    assert FL(one, 1, 3, 10, kq.STOP_ON_STABLE, None) == 1  # would synchronise per layer
    bad = [_job(1, n=0), _job(1, K=2048), _job(1, W=None), _job(1, ws=None),
           _job(1, levels=ctypes.c_void_p(1 << 24)),  # levels without codes
           _job(1, W_out=ctypes.c_void_p(1 << 24))]  # recovery without codes
    for j in bad:
        assert FL((kq.LayerJob * 1)(j), 1, 3, 10, 0, None) == 1
    two = (kq.LayerJob * 2)(_job(1), _job(2, ws=_job(1).ws))  # one workspace for two layers
    assert FL(two, 2, 3, 10, 0, None) == 1


def test_trace_arguments_checked_on_host(lib):
    assert lib.kq_trace_start(0) == 1
    assert lib.kq_trace_start((1 << 20) + 1) == 1
    name, ms = ctypes.c_char_p(), ctypes.c_float()
    assert lib.kq_trace_get(-1, ctypes.byref(name), ctypes.byref(ms)) == 1
    assert lib.kq_trace_get(lib.kq_trace_count(), ctypes.byref(name), ctypes.byref(ms)) == 1
    assert lib.kq_trace_stop() == 0


def test_cuda_failure_returns_status_without_device(lib):
    # Every argument valid, no CUDA device: the first CUDA runtime call fails, and the
    # entry point returns KQ_ERR_CUDA (4) before anything is enqueued. (Skipped where a
    # GPU exists: the placeholder pointers below must never reach a kernel.)
    import torch
    if torch.cuda.is_available():
        pytest.skip("a CUDA device is present")
    L = lib
    good = ctypes.c_void_p(1 << 20)
    ws_bytes = kq.kq_workspace_bytes(1024, 16)
    assert L.kq_assign(good, 1024, good, 16, None, good, None, good, ws_bytes, None) == 4
    assert L.kq_update_centroids(good, 1024, good, 16, good, good, good, good, ws_bytes, None) == 4
    assert L.kq_fit_codebook(good, 1024, 16, good, 3, 0, good, good, good, None, None, good, ws_bytes, None) == 4
    assert L.kq_quantize_codebook_6bit(good, 16, good, 10, good, good, None, good, ws_bytes, None) == 4
    assert L.kq_reconstruct(good, 1024, good, 16, None, None, good, good, ws_bytes, None) == 4
    assert L.kq_quantize_reconstruct(good, 1024, good, 16, good, None, good, good, ws_bytes, None) == 4
    assert L.kq_device_status(good, ws_bytes, None, None) == 4
    u64 = ctypes.c_uint64()
    assert L.kq_fit_prune_stats(good, ws_bytes, ctypes.byref(u64), ctypes.byref(u64), None) == 4
    assert L.kq_trace_start(4) == 4  # no device to make events on
    jobs = (kq.LayerJob * 2)(_job(1), _job(2))
    assert L.kq_fit_layers(jobs, 2, 3, 10, kq.FIT_PRUNE, None) == 4
