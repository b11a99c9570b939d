"""kq_fit_layers: every layer of a set through one call gives, bit for bit, what the
single-layer calls give (init, fit, 6-bit codebook quantisation, K+C recovery),
whatever internal stream a layer lands on."""
import numpy as np
import pytest
import torch

import synth
from gpu_util import dev, to_dev
from paper_2003_05148_gb300 import kq

pytestmark = pytest.mark.gpu


def _buffers(lay, T, with_sel=True, quantize=True, recover=True):
    W, sel = synth.layer_inputs(lay)
    n, K = W.shape[0], lay.K
    Wd = to_dev(W)
    b = {"W": Wd, "C": torch.empty(K, 9, dtype=torch.float32, device=dev()),
         "idx": torch.empty(n, dtype=torch.int32, device=dev()),
         "counts": torch.empty(K, dtype=torch.int32, device=dev()),
         "objective": torch.empty(T + 1, dtype=torch.float64, device=dev()),
         "ws": kq.workspace(n, K, dev())}
    if with_sel:
        b["sel"] = to_dev(sel)
    else:  # the caller's own C_0: the seeded rows, gathered on the host
        b["C"].copy_(torch.from_numpy(W[sel]))
    if quantize:
        b["levels"] = torch.empty(64, dtype=torch.float32, device=dev())
        b["codes"] = torch.empty(K, 9, dtype=torch.uint8, device=dev())
        if recover:
            b["W_out"] = torch.empty(n, 9, dtype=torch.float32, device=dev())
    return b


def _single(b, T, level_iters, flags):
    if "sel" in b:
        kq.kq_init_codebook(b["W"], b["sel"], b["C"], b["ws"])
    kq.kq_fit_codebook(b["W"], b["C"], T, b["C"], b["idx"], b["counts"], b["objective"], b["ws"], flags=flags)
    if "codes" in b:
        kq.kq_quantize_codebook_6bit(b["C"], b["counts"], level_iters, b["levels"], b["codes"], None, b["ws"])
    if "W_out" in b:
        kq.kq_reconstruct(b["idx"], None, b["codes"], b["levels"], b["W_out"], b["ws"], K=b["C"].shape[0])


def _outputs(b):
    return {k: v.cpu().numpy() for k, v in b.items() if k in ("C", "idx", "counts", "objective", "levels", "codes",
                                                                "W_out")}


@pytest.mark.parametrize("cfg,picks,flags", [
    (3, [0, 1, 2, 3, 4, 8], 0),      # VGG-16: one-launch small fits, K = 48 and 512 on both assign paths
    (4, [0, 4, 5, 9], 0),            # ResNet-18: K = 1024 .. 16384, hint order from 4096 on
    (4, [5, 6], kq.FIT_PRUNE),       # pruned tensor-core fits
])
def test_fit_layers_equals_single_layer_calls(cfg, picks, flags):
    wl = synth.workload(cfg)
    lays = [wl.layers[i] for i in picks]
    T, LI = 5, 60
    # variety: one layer starts from a given C_0, one stops after the fit, one skips the recovery
    opts = [dict(with_sel=(i != 1), quantize=(i != 2), recover=(i != 3)) for i in range(len(lays))]
    ref = []
    for lay, o in zip(lays, opts):
        b = _buffers(lay, T, **o)
        _single(b, T, LI, flags)
        ref.append(b)
    got = [_buffers(lay, T, **o) for lay, o in zip(lays, opts)]
    kq.kq_fit_layers(got, T, LI, flags)
    torch.cuda.synchronize()
    for i, (r, g) in enumerate(zip(ref, got)):
        assert kq.kq_device_status(r["ws"])[0] == 0 and kq.kq_device_status(g["ws"])[0] == 0
        ro, go = _outputs(r), _outputs(g)
        assert ro.keys() == go.keys()
        for k in ro:
            assert np.array_equal(ro[k].view(np.uint8), go[k].view(np.uint8)), (i, k)


def test_fit_layers_orders_against_the_callers_stream():
    # work enqueued on the caller's stream before the call is seen by every layer, and
    # work enqueued after it sees every layer's outputs
    lays = synth.workload(4).layers[:3]
    T = 3
    s = torch.cuda.Stream(device=dev())
    bufs = [_buffers(lay, T, with_sel=False) for lay in lays]
    ref = []
    for lay in lays:
        b = _buffers(lay, T, with_sel=False)
        _single(b, T, 30, 0)
        ref.append(_outputs(b))
    s.wait_stream(torch.cuda.current_stream())  # the buffers were filled there
    with torch.cuda.stream(s):
        C0 = [b["C"].clone() for b in bufs]
        for b in bufs:
            b["C"].zero_()  # overwritten below on the same stream, before the call
        for b, c in zip(bufs, C0):
            b["C"].copy_(c)
        kq.kq_fit_layers(bufs, T, 30, 0, stream=s)
        outs = [b["W_out"].clone() for b in bufs]  # after the call, on the same stream
    s.synchronize()
    for r, b, o in zip(ref, bufs, outs):
        assert np.array_equal(r["W_out"].view(np.uint8), o.cpu().numpy().view(np.uint8))
        assert np.array_equal(r["idx"], b["idx"].cpu().numpy())


def test_fit_layers_reports_a_failing_layer():
    # a layer whose workspace is too small fails with KQ_ERR_WORKSPACE; the call
    # still joins the streams it forked, so the caller's stream stays usable and the
    # layers enqueued before the failing one complete
    lays = synth.workload(4).layers[:3]
    T = 2
    bufs = [_buffers(lay, T, with_sel=False) for lay in lays]
    ref = []
    for lay in lays:
        b = _buffers(lay, T, with_sel=False)
        _single(b, T, 30, 0)
        ref.append(_outputs(b))
    bufs[2]["ws"] = bufs[2]["ws"][:4096]  # the smallest layer is dealt last: its fit fails
    with pytest.raises(kq.KQError) as err:
        kq.kq_fit_layers(bufs, T, 30, 0)
    assert err.value.status == 6  # KQ_ERR_WORKSPACE
    torch.cuda.current_stream().synchronize()
    for r, b in zip(ref[:2], bufs[:2]):
        assert np.array_equal(r["idx"], b["idx"].cpu().numpy())
        assert np.array_equal(r["W_out"].view(np.uint8), b["W_out"].cpu().numpy().view(np.uint8))
