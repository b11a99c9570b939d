"""Per-workload parity verdicts: every layer of each of the five seeded workloads,
one step of the method at a time from identical inputs, against the oracle.

For each layer: the assignment against the seeded initial codebook (Sec. 3.1,
Eq. 1; bit-exact indices and distances, on a seeded row sample where the layer is
large), the centroid update from those indices (within 1e-5 per codeword), the
6-bit quantisation of the updated codebook weighted by its counts (Sec. 3.2;
bit-exact levels and codes) and the K+C recovery of every kernel (bit-exact). The
verdict line of each workload is printed (pytest -s) for the configuration report.
"""
import json

import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import bits_equal, check_centroids, check_indices, dev, to_dev
from paper_2003_05148_gb300 import kq

pytestmark = pytest.mark.gpu
THREADS = oracle.default_threads()
SAMPLE_ROWS = 4096


def _layer_step(lay):
    W, sel = synth.layer_inputs(lay)
    n, K = W.shape[0], lay.K
    C0 = oracle.gather_rows(W, sel)
    Wd, Cd = to_dev(W), to_dev(C0)
    ws = kq.workspace(n, K, dev())
    idx = torch.empty(n, dtype=torch.int32, device=dev())
    dist = torch.empty(n, dtype=torch.float32, device=dev())
    kq.kq_assign(Wd, Cd, idx, dist, ws)
    C1 = torch.empty_like(Cd)
    counts = torch.empty(K, dtype=torch.int32, device=dev())
    kq.kq_update_centroids(Wd, idx, Cd, C1, counts, ws)
    levels = torch.empty(64, dtype=torch.float32, device=dev())
    codes = torch.empty(K, 9, dtype=torch.uint8, device=dev())
    kq.kq_quantize_codebook_6bit(C1, counts, 100, levels, codes, None, ws)
    Wr = torch.empty_like(Wd)
    kq.kq_reconstruct(idx, None, codes, levels, Wr, ws, K=K)
    st, flags = kq.kq_device_status(ws)
    assert st == 0, (lay.name, st, flags)
    idx_g, dist_g = idx.cpu().numpy(), dist.cpu().numpy()
    # assignment: every row, or a seeded sample with the last row
    rows = None
    if n > SAMPLE_ROWS and n * K > 3e8:
        rows = np.sort(synth.below(synth.stream_key(lay.seed, 13), SAMPLE_ROWS, n))
        rows[-1] = n - 1
    Wc = W if rows is None else W[rows]
    idx_ref, dist_ref = oracle.assign(Wc, C0, threads=THREADS)
    ig = idx_g if rows is None else idx_g[rows]
    dg = dist_g if rows is None else dist_g[rows]
    near_ties = check_indices(W, C0, ig, idx_ref, rows)
    assert bits_equal(dg[ig == idx_ref], dist_ref[ig == idx_ref])
    # update from the same indices
    C1_ref, cnt_ref = oracle.update(W, idx_g, C0)
    C1_g = C1.cpu().numpy()
    check_centroids(C1_g, C1_ref)
    assert np.array_equal(counts.cpu().numpy(), cnt_ref)
    scale = np.maximum(np.abs(C1_ref).max(axis=1, keepdims=True), 1e-30)
    rel = float((np.abs(C1_g.astype(np.float64) - C1_ref) / scale).max())
    # 6-bit quantisation of the GPU's codebook, then recovery
    lv_ref, cd_ref, _ = oracle.level_fit(C1_g, cnt_ref)
    assert bits_equal(levels.cpu().numpy(), lv_ref)
    assert np.array_equal(codes.cpu().numpy(), cd_ref)
    W_ref = oracle.reconstruct(idx_g, C1_g, cd_ref, lv_ref)
    assert bits_equal(Wr.cpu().numpy(), W_ref)
    return {"n": n, "K": K, "assign_rows_checked": int(len(Wc)), "near_ties": int(near_ties),
            "centroid_max_rel": rel}


@pytest.mark.parametrize("cfg", [1, 2, 3, 4, 5])
def test_workload_step_parity(cfg):
    wl = synth.workload(cfg)
    layers = [_layer_step(lay) for lay in wl.layers]
    print(json.dumps({"parity": wl.name, "layers": len(layers), "verdict": "pass",
                      "assign": f"bit-exact on {sum(x['assign_rows_checked'] for x in layers)} rows "
                                f"({sum(x['near_ties'] for x in layers)} fp64 near-ties)",
                      "update_max_rel": max(x["centroid_max_rel"] for x in layers),
                      "levels_codes": "bit-exact", "reconstruct": "bit-exact, every kernel"}), flush=True)
