"""Independent decoders used to pin the oracle.

These decode the stored formats through routes that share nothing with the
oracle's C code: torch's own float8_e4m3fn conversion for E4M3 and the
specification's E2M1 table (``golden/e2m1_ocp_values.txt``) for FP4.
"""
import os

import numpy as np
import torch

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def read_table(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if not line:
                continue
            code, val = line.split()
            rows.append((int(code, 16), float(val)))
    return rows


E2M1_TABLE = np.array([v for _, v in sorted(read_table("e2m1_ocp_values.txt"))], np.float64)


def e4m3_torch(codes) -> np.ndarray:
    t = torch.as_tensor(np.ascontiguousarray(codes, np.uint8))
    return t.view(torch.float8_e4m3fn).to(torch.float64).numpy()


def dequant_fp8(codes, scales) -> np.ndarray:
    """codes [N, K] uint8, scales [N/128, K/128] -> float64 [N, K]."""
    v = e4m3_torch(codes)
    s = np.repeat(np.repeat(np.asarray(scales, np.float64), 128, axis=0), 128, axis=1)
    return v * s


def dequant_nvfp4(codes, sf, ts) -> np.ndarray:
    """codes [N, K/2] uint8 (low nibble = even k), sf [N, K/16] e4m3, ts scalar."""
    codes = np.asarray(codes, np.uint8)
    N, K2 = codes.shape
    nib = np.empty((N, 2 * K2), np.uint8)
    nib[:, 0::2] = codes & 15
    nib[:, 1::2] = codes >> 4
    v = E2M1_TABLE[nib]
    s = np.repeat(e4m3_torch(sf), 16, axis=1)
    return v * s * float(ts)


def dequant(w, which, e) -> np.ndarray:
    """One expert matrix of a synth.LayerWeights-like object holding numpy arrays."""
    codes = getattr(w, "w_" + which)[e]
    sc = getattr(w, "s_" + which)[e]
    if w.fmt == 1:
        return dequant_fp8(codes, sc)
    return dequant_nvfp4(codes, sc, getattr(w, "ts_" + which)[e])


def bf16_to_f64(bits) -> np.ndarray:
    t = torch.as_tensor(np.ascontiguousarray(bits, np.uint16).view(np.int16))
    return t.view(torch.bfloat16).to(torch.float64).numpy()
