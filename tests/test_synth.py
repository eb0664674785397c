"""The synthetic-input generator: determinism and encoder behaviour."""
import numpy as np
import torch

from paper_2609_11133_gb300 import synth
from tests import indep


def test_generators_are_deterministic():
    a = synth.make_weights(2, 2, 64, 32, seed=3)
    b = synth.make_weights(2, 2, 64, 32, seed=3)
    for x, y in zip(a.tensors(), b.tensors()):
        assert torch.equal(x, y)
    assert torch.equal(synth.make_x(3, 64, seed=1), synth.make_x(3, 64, seed=1))
    assert not torch.equal(synth.make_x(3, 64, seed=1), synth.make_x(3, 64, seed=2))


def test_e2m1_encoder_rounds_to_nearest_even():
    vals = torch.tensor([0.0, 0.25, 0.26, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0, 5.1, 7.0, -0.75, -0.0])
    codes = synth.encode_e2m1(vals)
    dec = indep.E2M1_TABLE[codes.numpy()]
    assert list(dec) == [0.0, 0.0, 0.5, 1.0, 1.0, 2.0, 2.0, 4.0, 4.0, 6.0, 6.0, -1.0, -0.0]


def test_fp8_block_quantiser_hits_the_amax():
    w = torch.randn(256, 384) * 0.02
    codes, scales = synth.quantize_fp8_block(w)
    assert scales.shape == (2, 3)
    deq = torch.tensor(indep.dequant_fp8(codes.numpy(), scales.numpy()))
    blk = deq.reshape(2, 128, 3, 128).abs().amax(dim=(1, 3))
    ref = w.reshape(2, 128, 3, 128).abs().amax(dim=(1, 3)).double()
    assert torch.allclose(blk, ref, rtol=1e-6)
    assert (deq - w.double()).abs().max() <= scales.max() * 16  # within half an e4m3 step at 448


def test_nvfp4_quantiser_error_is_bounded():
    w = torch.randn(64, 128) * 0.02
    codes, sf, ts = synth.quantize_nvfp4(w)
    deq = indep.dequant_nvfp4(codes.numpy(), sf.numpy(), ts)
    err = np.abs(deq - w.double().numpy())
    # per 16-block the step of e2m1 at the top is 2 units of sf*ts
    step = np.repeat(indep.e4m3_torch(sf.numpy()) * ts, 16, axis=1)
    assert (err <= step * 1.0 + 1e-12).all()
