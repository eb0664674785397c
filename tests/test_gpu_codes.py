"""Every weight code through the device decoders, one code per token.

The layer is set up so that token p's output depends on one stored code and nothing else:
- one expert (E = 1, k = 1, gate 1);
- token p is one-hot on column p;
- in that column, gate and up have a single nonzero entry, in row i_p: the gate entry is the
  constant 2.0 and the up entry is the code under test;
- the down matrix is the identity.
Then out[p, i_p] = silu(2) * dec(code_p) and every other output is zero.

Every activation row (x, and h after SwiGLU) has a single nonzero element, so the GPU's
activation terms represent it exactly.  An output within 2^-7 of the format's value shows that the
device decoded that code (and, for NVFP4, its block scale) correctly.  A wrong decode is off by at
least 1/15: that is the smallest relative step between neighbouring E4M3 or UE4M3 magnitudes, and
the E2M1 steps are larger.

- FP8: all 254 E4M3 codes (0x7F and 0xFF are NaN and never stored).
- NVFP4: all 16 E2M1 codes under each of the 127 UE4M3 block scales 0x00-0x7E.

The tensor-core engines run in this process.  The warp-MMA engine, which decodes on the CUDA
cores, runs the same cases in a subprocess.  The oracle's decoders are pinned to the OCP tables in
the CPU tests."""
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2609_11133_gb300 import synth
from tests.gpu_harness import Case

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
REL = 2.0 ** -7
SILU2 = 2.0 / (1.0 + np.exp(-2.0))

E4M3_ONE, E4M3_TWO = 0x38, 0x40
E2M1_ONE, E2M1_TWO = 2, 4


def _one_hot_x(T, H, device):
    x = torch.zeros((T, H), dtype=torch.bfloat16)
    x[torch.arange(T), torch.arange(T)] = 1.0
    return x.to(device)


def fp8_case(device="cuda"):
    """Token p (one per non-NaN E4M3 code): up[p, p] = code_p, gate[p, p] = 2.0."""
    codes = [c for c in range(256) if (c & 0x7F) != 0x7F]
    T, H, I = len(codes), 256, 256
    wg = torch.zeros((1, I, H), dtype=torch.uint8)
    wu = torch.zeros((1, I, H), dtype=torch.uint8)
    wd = torch.zeros((1, H, I), dtype=torch.uint8)
    for p, c in enumerate(codes):
        wu[0, p, p] = c
        wg[0, p, p] = E4M3_TWO
    for j in range(I):
        wd[0, j, j] = E4M3_ONE
    ones = lambda n, k: torch.ones((1, n // 128, k // 128), dtype=torch.float32, device=device)
    w = synth.LayerWeights(synth.FMT_FP8, 1, H, I, wg.to(device), wu.to(device), wd.to(device),
                           ones(I, H), ones(I, H), ones(H, I))
    expect = [(p, p, SILU2 * oracle.e4m3(c)) for p, c in enumerate(codes)]
    return w, _one_hot_x(T, H, device), expect


def nvfp4_case(device="cuda"):
    """Token p = 16 s + c (c: E2M1 code, s: UE4M3 block scale 0x00-0x7E) is one-hot
    on column p; up row p % 256 holds code c there under block scale s."""
    pairs = [(c, s) for s in range(0x7F) for c in range(16)]
    T, H, I = len(pairs), 2048, 256
    wg = torch.zeros((1, I, H // 2), dtype=torch.uint8)
    wu = torch.zeros((1, I, H // 2), dtype=torch.uint8)
    wd = torch.zeros((1, H, I // 2), dtype=torch.uint8)
    sg = torch.zeros((1, I, H // 16), dtype=torch.uint8)
    su = torch.zeros((1, I, H // 16), dtype=torch.uint8)
    sd = torch.zeros((1, H, I // 16), dtype=torch.uint8)
    expect = []
    for p, (c, s) in enumerate(pairs):
        i, sh = p % I, 4 * (p % 2)  # element p: byte p / 2, low nibble if even
        # (row i, block p / 16) is a different scale cell for every p < 16 * I
        wu[0, i, p // 2] |= c << sh
        su[0, i, p // 16] = s
        wg[0, i, p // 2] |= E2M1_TWO << sh
        sg[0, i, p // 16] = E4M3_ONE
        expect.append((p, i, SILU2 * oracle.e2m1(c) * oracle.e4m3(s)))
    for j in range(I):
        wd[0, j, j // 2] |= E2M1_ONE << (4 * (j % 2))
        sd[0, j, j // 16] = E4M3_ONE
    ts = lambda: torch.ones((1,), dtype=torch.float32, device=device)
    w = synth.LayerWeights(synth.FMT_NVFP4, 1, H, I, wg.to(device), wu.to(device), wd.to(device),
                           sg.to(device), su.to(device), sd.to(device), ts(), ts(), ts())
    return w, _one_hot_x(T, H, device), expect


def _check(fmt):
    w, x, expect = fp8_case() if fmt == 1 else nvfp4_case()
    T, H = x.shape
    wr = torch.zeros((1, H), dtype=torch.float32, device="cuda")
    c = Case(fmt, T=T, H=H, E=1, k=1, I=w.I, w=w, wr=wr, x=x).run()
    ref = c.reference()
    got = c.out.float().cpu().numpy().astype(np.float64)
    want = np.zeros_like(ref)
    for p, i, v in expect:
        want[p, i] = v
    # the oracle reads the stored codes as the formats define them ...
    assert np.allclose(ref, want, rtol=1e-14, atol=0.0)
    # ... and so does the device, code by code
    ok = np.abs(got - want) <= REL * np.abs(want)
    bad = np.argwhere(~ok)
    assert ok.all(), f"{len(bad)} outputs off, first {bad[:5].tolist()}: " \
                     f"got {got[tuple(bad[0])]} want {want[tuple(bad[0])]}"


@pytest.mark.parametrize("fmt", [1, 2])
def test_every_code_decodes_on_the_tensor_cores(fmt):
    _check(fmt)


SCRIPT = r"""
import sys
sys.path.insert(0, {root!r})
from tests.test_gpu_codes import _check
_check(1)
_check(2)
print("CODES_OK")
"""


def test_every_code_decodes_in_the_warp_mma_engine():
    env = dict(os.environ, MOE_ENGINE="mma")
    r = subprocess.run([sys.executable, "-c", SCRIPT.format(root=ROOT)], env=env,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0 and "CODES_OK" in r.stdout, r.stdout[-2000:] + r.stderr[-4000:]
