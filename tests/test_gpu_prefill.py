"""Prefill-shaped batches through the decode layer: thousands of tokens per call.

Every expert then holds a hundred or more tokens, so its items come in many chunks (16 tokens for
NVFP4, 32 for FP8).  The chunks of one row tile run one after another and re-read the expert's
weight tile from L2.  The activation terms are gathered into compact rows first (more than 64
tokens).  The routing is checked for every token, the output on sampled tokens."""
import numpy as np
import pytest

from tests.gpu_harness import Case

pytestmark = pytest.mark.gpu

FP8, FP4 = 1, 2


def test_qwen3_235b_nvfp4_prefill_sampled_tokens():
    c = Case(FP4, T=2048, H=4096, E=128, k=8, I=1536, seed=3).run()
    n = np.bincount(c.ids.cpu().numpy().reshape(-1), minlength=128)
    assert n.min() >= 64  # every expert spans several 16-token chunks
    c.check_output(tokens=[0, 511, 1024, 1537, 2047])


def test_fp8_prefill_sampled_tokens():
    # the 480B layer's expert shape with 40 experts: about 410 tokens each
    c = Case(FP8, T=2048, H=6144, E=40, k=8, I=2560, seed=4).run()
    n = np.bincount(c.ids.cpu().numpy().reshape(-1), minlength=40)
    assert n.min() >= 128
    c.check_output(tokens=[0, 777, 2047])
