"""The seeded input generator: published SplitMix64 outputs, determinism, shapes."""
import numpy as np
import pytest

import synth


def test_splitmix64_reference_outputs():
    # First outputs of SplitMix64 seeded with 0 (Steele, Lea, Flood 2014).
    got = [int(x) for x in synth.u64(np.uint64(0), 0, 3)]
    assert got == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]
    # counter evaluation: a window equals the same positions of a longer run
    k = synth.stream_key(7, 3)
    assert np.array_equal(synth.u64(k, 5, 10), synth.u64(k, 0, 15)[5:])


def test_uniform_and_normal_moments():
    u = synth.uniform01(synth.stream_key(1, 1), 0, 200000)
    assert u.min() > 0 and u.max() < 1
    assert abs(u.mean() - 0.5) < 0.01
    z = synth.normal(synth.stream_key(2, 1), 200001)
    assert z.shape == (200001,)
    assert abs(z.mean()) < 0.01 and abs(z.std() - 1) < 0.01


@pytest.mark.parametrize("cfg", [1, 2])
def test_layer_inputs_deterministic(cfg):
    lay = synth.workload(cfg).layers[0]
    W1, s1 = synth.layer_inputs(lay)
    W2, s2 = synth.layer_inputs(lay)
    assert W1.dtype == np.float32 and W1.shape == (lay.n, 9)
    assert np.array_equal(W1, W2) and np.array_equal(s1, s2)
    assert len(set(s1.tolist())) == lay.K and s1.min() >= 0 and s1.max() < lay.n
    # Gaussian mixture: total std = sigma * sqrt(1 + 0.3^2)
    assert abs(W1.std() / (lay.sigma * np.sqrt(1.09)) - 1) < 0.1


def test_init_selection_full_permutation():
    s = synth.init_selection(50, 50, 9)
    assert sorted(s.tolist()) == list(range(50))


def test_workload_shapes():
    w3 = synth.workload(3)
    assert len(w3.layers) == 13 and sum(l.n for l in w3.layers) == 1634496
    assert w3.layers[0].K == 48 and all(l.K == 512 for l in w3.layers[1:])
    w4 = synth.workload(4)
    assert len(w4.layers) == 16 and sum(l.n for l in w4.layers) == 1220608
    assert max(l.K for l in w4.layers) == 16384
    w5 = synth.workload(5)
    assert w5.layers[0].n == 4194304 and w5.layers[0].K == 65536 and w5.iters == 10
