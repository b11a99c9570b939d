"""GPU parity of Algorithm 1 (adaptive codebook size, Eq. 3) against the oracle's
search on the same seeded layers: the same sizes tested in the same order, the
same result, errors equal up to the order of the objective sums."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import bits_equal, dev, to_dev
from paper_2003_05148_gb300 import kq

pytestmark = pytest.mark.gpu


def gpu_search(W, sel, alpha, r, steps, iters):
    n = W.shape[0]
    n_init = oracle.initial_size(n, alpha)
    C = torch.empty(n_init, 9, dtype=torch.float32, device=dev())
    idx = torch.empty(n, dtype=torch.int32, device=dev())
    counts = torch.empty(n_init, dtype=torch.int32, device=dev())
    ws = kq.workspace(n, n_init, dev())
    k, err, trace = kq.kq_search_codebook_size(to_dev(W), to_dev(sel), alpha, r, steps, iters, C, idx, counts, ws)
    st, _ = kq.kq_device_status(ws)
    return k, err, trace, C[:k].cpu().numpy(), idx.cpu().numpy(), counts[:k].cpu().numpy(), st


@pytest.mark.parametrize("cfg,alpha,r,steps,iters", [(1, 0.25, 0.5, 8, 3), (1, 0.1, 0.0, 6, 5), (2, 0.05, 0.5, 6, 2)])
def test_search_matches_oracle(cfg, alpha, r, steps, iters):
    lay = synth.workload(cfg).layers[0]
    W, _ = synth.layer_inputs(lay)
    n = W.shape[0]
    sel = synth.init_selection(n, oracle.initial_size(n, alpha), lay.seed + 1)
    k_g, e_g, tr_g, C_g, idx_g, cnt_g, st = gpu_search(W, sel, alpha, r, steps, iters)
    k_r, tr_r = oracle.search_codebook_size(W, sel, alpha, r, steps, iters, threads=oracle.default_threads())
    assert st == 0
    # every decision clears the target by far more than summation-order rounding
    e_target = tr_r[0][1] * (1 + r)
    assert all(abs(e - e_target) > 1e-9 * e_target for _, e in tr_r[1:])
    assert [s for s, _ in tr_g] == [s for s, _ in tr_r] and k_g == k_r
    for (_, a), (_, b) in zip(tr_g, tr_r):
        assert abs(a - b) <= 1e-12 + 1e-9 * b
    # the outputs are the fit of the chosen size
    C_r, idx_r, cnt_r, _ = oracle.fit(W, oracle.gather_rows(W, sel[:k_r]), iters, threads=oracle.default_threads())
    assert np.array_equal(idx_g, idx_r) and np.array_equal(cnt_g, cnt_r)
    assert np.abs(C_g - C_r).max() <= 1e-5 * np.abs(C_r).max()
    assert dict(tr_g).get(k_g, e_g) == e_g


def test_search_zero_steps_keeps_initial_size():
    lay = synth.workload(1).layers[0]
    W, _ = synth.layer_inputs(lay)
    sel = synth.init_selection(W.shape[0], 409, lay.seed + 1)
    k, err, trace, _, _, _, st = gpu_search(W, sel, 0.1, 0.5, 0, 2)
    assert st == 0 and k == 409 and trace == [(409, err)]
