"""The chained linear path of a decoder block (QKV -> V slice -> out ->
fc1 + ReLU -> fc2, each layer calibrated on the activations it receives)
against the oracle running the same chain on its own outputs.  With the
epilogue defined as one fp32 fma rounded to fp16, every layer's codes,
parameters and outputs match bit for bit, so the chain cannot drift."""
import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


def _oracle_chain(x_cal, x, weights, h, bits, cols=None):
    """Per layer: (mn, mx, z, s, r, qw, sw, bf, y) following the block's data flow."""
    out = []
    acts_cal, acts = x_cal, x
    for i, (w, b) in enumerate(weights):
        mn, mx = oracle.calibrate(acts_cal)
        z, s, r = oracle.params(mn, mx, bits)
        qw, sw, bf = oracle.fold(w, b, z, s, bits)
        relu = i == 2
        _, _, y = oracle.linear(acts, qw, sw, bf, z, r, bits, relu)
        out.append(dict(mn=mn, mx=mx, z=z, s=s, r=r, qw=qw, sw=sw, bf=bf, y=y))
        if i < 3:
            _, _, yc = oracle.linear(acts_cal, qw, sw, bf, z, r, bits, relu)
            acts_cal = yc[:, 2 * h:].copy() if i == 0 else yc
            acts = y[:, 2 * h:].copy() if i == 0 else y
    return out


def _check(block, x_cal, x, weights, h, bits):
    from paper_2406_18832_gb300 import binding
    block.calibrate(x_cal.cuda(), [(w.cuda(), b.cuda()) for w, b in weights])
    outs = block.forward(x.cuda())
    torch.cuda.synchronize()
    assert binding.ot_get_device_status() == binding.OT_OK
    ref = _oracle_chain(x_cal.numpy(), x.numpy(), [(w.numpy(), b.numpy()) for w, b in weights], h, bits)
    names = ("qkv", "o", "f", "y")
    for i, (ql, name) in enumerate(zip(block.layers, names)):
        r = ref[i]
        for k, t in (("mn", ql.ch_min), ("mx", ql.ch_max), ("z", ql.z), ("s", ql.s), ("r", ql.r),
                     ("sw", ql.sw), ("bf", ql.b_fold)):
            assert np.array_equal(t.cpu().numpy(), r[k]), (name, k)
        assert np.array_equal(ql.qw.cpu().numpy(), r["qw"]), (name, "qw")
        y = outs[name].cpu().numpy()
        assert np.array_equal(y.astype(np.float32), r["y"].astype(np.float32)), name
    assert (outs["f"] >= 0).all()


@pytest.mark.parametrize("bits", [8, 6])
def test_small_block_chain(bits):
    from paper_2406_18832_gb300 import QuantizedBlockLinears, synth
    h, ffn, T, M = 512, 2048, 256, 64
    lay = synth.Layer("qkv", h, 3 * h, 0.01)
    x_cal = synth.activations(9, 0, lay, T, 3)
    x = synth.activations(9, 0, lay, M, 4)
    shapes = [(h, 3 * h), (h, h), (h, ffn), (ffn, h)]
    weights = [synth.weights(9, i, synth.Layer("l", K, N)) for i, (K, N) in enumerate(shapes)]
    _check(QuantizedBlockLinears(h, ffn, bits, bits), x_cal, x, weights, h, bits)


@pytest.mark.parametrize("bits", [8, 6])
def test_opt30b_block_chain_full_width(bits):
    """Config-5 widths (hidden 7168, FFN 28672) with few tokens so that the
    oracle can run the whole chain, calibration included."""
    from paper_2406_18832_gb300 import QuantizedBlockLinears, synth
    c = synth.CONFIGS[5]
    h, ffn = 7168, 28672
    x_cal = synth.activations(5, 0, c.layers[0], 16, 3)
    x = synth.activations(5, 0, c.layers[0], 4, 4)
    weights = [synth.weights(5, i, layer) for i, layer in enumerate(c.layers)]
    _check(QuantizedBlockLinears(h, ffn, bits, bits), x_cal, x, weights, h, bits)
