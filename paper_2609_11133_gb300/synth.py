"""Seeded synthetic inputs for the MoE decode layer.

This module only draws random numbers and stores them in the layer's input
formats (bf16 activations, fp32 router, FP8/NVFP4 expert weights).  It holds
none of the layer's arithmetic: it never decodes a weight, never routes a
token and never multiplies a matrix.  The CUDA path and the oracle both
consume exactly the tensors built here.

The shapes follow the MoE layers of the models the paper serves (Section 4,
"Setup": Qwen3-Coder-480B in FP8 and Qwen3-235B-A22B in NVFP4):

* activations x[T, H]: N(0, 1) rounded to bf16;
* router Wr[E, H]: N(0, 0.02) in fp32;
* expert matrices: N(0, 0.02) quantised to
  - FP8: E4M3 codes with one fp32 scale per 128x128 tile, scale = amax/448,
    code = round-to-nearest-even(w / scale) (saturating at 448);
  - NVFP4: E2M1 codes (two per byte, low nibble = even K) with one E4M3
    scale per 16 elements along K and one fp32 scale per expert matrix:
    ts = amax/(448*6), sf = e4m3(amax16/(6*ts)), code = e2m1_rne(w/(sf*ts)).

Everything is generated with ``torch`` on the requested device, expert by
expert, so that the 7 GB FP8 layer builds in seconds on the GPU.
"""
from __future__ import annotations

import math
from dataclasses import dataclass
from typing import Optional

import torch

FMT_FP8 = 1
FMT_NVFP4 = 2

_E4M3_MAX = 448.0
_E2M1_MAX = 6.0
# decision points between consecutive E2M1 magnitudes {0,.5,1,1.5,2,3,4,6}
_E2M1_MIDS = (0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0)


def _gen(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) & 0x7FFFFFFFFFFFFFFF)
    return g


def _normal(shape, std, device, seed) -> torch.Tensor:
    return torch.randn(shape, generator=_gen(device, seed), device=device,
                       dtype=torch.float32) * std


# ----------------------------------------------------------------- encoders
def encode_e4m3(v: torch.Tensor) -> torch.Tensor:
    """fp32 -> E4M3 code bytes (round to nearest even, saturating at +-448)."""
    return v.clamp(-_E4M3_MAX, _E4M3_MAX).to(torch.float8_e4m3fn).view(torch.uint8)


def encode_e2m1(v: torch.Tensor) -> torch.Tensor:
    """fp32 -> 4-bit E2M1 codes in uint8 (round to nearest even, saturating at +-6)."""
    mag = v.abs().clamp(max=_E2M1_MAX)
    mids = torch.tensor(_E2M1_MIDS, device=v.device, dtype=torch.float32)
    code = torch.bucketize(mag, mids, right=False)  # number of mids strictly below
    at_mid = (code < len(_E2M1_MIDS)) & (mids[code.clamp(max=len(_E2M1_MIDS) - 1)] == mag)
    code = code + (at_mid & (code % 2 == 1)).to(code.dtype)  # ties go to the even code
    sign = torch.signbit(v).to(torch.int64) << 3
    return (code | sign).to(torch.uint8)


def quantize_fp8_block(w: torch.Tensor):
    """w [N, K] fp32 -> (codes uint8 [N, K], scales fp32 [N/128, K/128])."""
    N, K = w.shape
    blk = w.reshape(N // 128, 128, K // 128, 128)
    amax = blk.abs().amax(dim=(1, 3))
    scale = torch.where(amax > 0, amax / _E4M3_MAX, torch.ones_like(amax))
    codes = encode_e4m3(blk / scale[:, None, :, None]).reshape(N, K)
    return codes, scale.contiguous()


def quantize_nvfp4(w: torch.Tensor):
    """w [N, K] fp32 -> (codes uint8 [N, K/2], sf uint8 [N, K/16], ts float)."""
    codes, sf, ts = _quantize_nvfp4(w)
    return codes, sf, float(ts)


def _quantize_nvfp4(w: torch.Tensor):
    """quantize_nvfp4 with the tensor scale left as a 0-d fp32 tensor on w's
    device (no host synchronisation)."""
    N, K = w.shape
    amax = w.abs().amax()
    ts = torch.where(amax > 0, amax / (_E4M3_MAX * _E2M1_MAX), torch.ones_like(amax))
    blk = w.reshape(N, K // 16, 16)
    bmax = blk.abs().amax(dim=2)
    sf_code = encode_e4m3(bmax / (_E2M1_MAX * ts))
    sf_val = sf_code.view(torch.float8_e4m3fn).to(torch.float32)
    denom = (sf_val * ts)[:, :, None]
    q = torch.where(denom > 0, blk / torch.where(denom > 0, denom, torch.ones_like(denom)),
                    torch.zeros_like(blk))
    nib = encode_e2m1(q).reshape(N, K)
    codes = (nib[:, 0::2] | (nib[:, 1::2] << 4)).contiguous()
    return codes, sf_code.contiguous(), ts


# ----------------------------------------------------------------- layer inputs
@dataclass
class LayerWeights:
    fmt: int
    E: int
    H: int
    I: int
    w_gate: torch.Tensor
    w_up: torch.Tensor
    w_down: torch.Tensor
    s_gate: torch.Tensor
    s_up: torch.Tensor
    s_down: torch.Tensor
    ts_gate: Optional[torch.Tensor] = None
    ts_up: Optional[torch.Tensor] = None
    ts_down: Optional[torch.Tensor] = None

    def nbytes_expert(self) -> int:
        """Stored bytes of one expert (codes + scales of the three matrices)."""
        tot = 0
        for t in (self.w_gate, self.w_up, self.w_down, self.s_gate, self.s_up, self.s_down):
            tot += t[0].numel() * t.element_size()
        if self.fmt == FMT_NVFP4:
            tot += 3 * 4
        return tot

    def tensors(self):
        return [t for t in (self.w_gate, self.w_up, self.w_down, self.s_gate, self.s_up,
                            self.s_down, self.ts_gate, self.ts_up, self.ts_down) if t is not None]

    def to(self, device) -> "LayerWeights":
        """A copy with every tensor on `device` (one copy per tensor)."""
        mv = lambda t: None if t is None else t.to(device)
        return LayerWeights(self.fmt, self.E, self.H, self.I, mv(self.w_gate), mv(self.w_up),
                            mv(self.w_down), mv(self.s_gate), mv(self.s_up), mv(self.s_down),
                            mv(self.ts_gate), mv(self.ts_up), mv(self.ts_down))


def make_weights(fmt: int, E: int, H: int, I: int, seed: int = 0, device="cpu",
                 std: float = 0.02, experts=None) -> LayerWeights:
    """Quantised expert weights of one layer, drawn expert by expert.

    ``experts``: optional subset of expert ids to draw (each expert has its own
    seed, so a subset equals the same rows of the full layer); the others are
    left zero.
    """
    dev = torch.device(device)
    todo = range(E) if experts is None else sorted(set(int(e) for e in experts))

    def one(which: int, N: int, K: int):
        if fmt == FMT_FP8:
            codes = torch.zeros((E, N, K), dtype=torch.uint8, device=dev)
            scales = torch.ones((E, N // 128, K // 128), dtype=torch.float32, device=dev)
            for e in todo:
                w = _normal((N, K), std, dev, seed * 1_000_003 + which * 10_007 + e)
                c, s = quantize_fp8_block(w)
                codes[e].copy_(c)
                scales[e].copy_(s)
            return codes, scales, None
        codes = torch.zeros((E, N, K // 2), dtype=torch.uint8, device=dev)
        sf = torch.zeros((E, N, K // 16), dtype=torch.uint8, device=dev)
        ts = torch.ones((E,), dtype=torch.float32, device=dev)
        for e in todo:
            w = _normal((N, K), std, dev, seed * 1_000_003 + which * 10_007 + e)
            c, s, t = _quantize_nvfp4(w)
            codes[e].copy_(c)
            sf[e].copy_(s)
            ts[e].copy_(t)
        return codes, sf, ts

    wg, sg, tg = one(1, I, H)
    wu, su, tu = one(2, I, H)
    wd, sd, td = one(3, H, I)
    return LayerWeights(fmt, E, H, I, wg, wu, wd, sg, su, sd, tg, tu, td)


def make_x(T: int, H: int, seed: int = 0, device="cpu", std: float = 1.0) -> torch.Tensor:
    """Activations x[T, H] ~ N(0, std^2) in bf16."""
    return _normal((T, H), std, torch.device(device), seed * 7_919 + 11).to(torch.bfloat16)


def make_router(E: int, H: int, seed: int = 0, device="cpu", std: float = 0.02) -> torch.Tensor:
    """Router rows Wr[E, H] ~ N(0, std^2) in fp32."""
    return _normal((E, H), std, torch.device(device), seed * 7_919 + 23)


def make_zipf_bias(E: int, H: int, s: float = 1.1, seed: int = 0, device="cpu",
                   router_std: float = 0.02) -> torch.Tensor:
    """Router bias that skews expert popularity towards Zipf(s).

    Expert of popularity rank r (a seeded random permutation of 1..E) gets
    b = -s * ln(r) * beta, beta = sigma_l * sqrt(6) / pi, with sigma_l the
    logit standard deviation of N(0,1) activations against N(0, router_std^2)
    rows.  With Gumbel logit noise of scale beta this is exactly Zipf(s) for
    the first choice; with the actual (normal) logits it is an approximation,
    so the realised popularity is measured, not assumed.
    """
    g = _gen("cpu", seed * 7_919 + 37)
    rank = torch.randperm(E, generator=g).to(torch.float64) + 1.0
    sigma_l = router_std * math.sqrt(H)
    beta = sigma_l * math.sqrt(6.0) / math.pi
    return (-s * torch.log(rank) * beta).to(torch.float32).to(device)


# ----------------------------------------------------------------- named workloads
# The layer shapes of the two models the paper serves, plus the small case.
WORKLOADS = {
    "tiny_fp8": dict(fmt=FMT_FP8, H=512, E=8, k=2, I=256),
    "qwen3_235b_nvfp4": dict(fmt=FMT_NVFP4, H=4096, E=128, k=8, I=1536),
    "qwen3_480b_fp8": dict(fmt=FMT_FP8, H=6144, E=160, k=8, I=2560),
}
