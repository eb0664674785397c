"""Helpers of the GPU parity tests: build seeded inputs on the device, run the
CUDA layer through the C ABI, and compute the float64 oracle on the host from
the very same stored tensors."""
import numpy as np
import torch

from oracle import oracle
from paper_2609_11133_gb300 import binding, synth
from tests.util_np import np_, oracle_weights

REL_TOL = 2e-2  # max|gpu - ref| <= REL_TOL * max|ref| per layer output
GATE_TOL = 1e-6


class Case:
    """One layer call.  Weights, router, input and residual are drawn from
    `seed` unless given (w, wr, x: device tensors; residual: True to draw one,
    or a [T, H] bf16 device tensor); `ow` is the oracle's copy of w, if the
    caller already made one."""

    def __init__(self, fmt, T, H, E, k, I, seed=0, bias=None, residual=False, flags=0,
                 w=None, wr=None, x=None, ow=None):
        dev = "cuda"
        self.fmt, self.T, self.H, self.E, self.k, self.I, self.flags = fmt, T, H, E, k, I, flags
        self.w = synth.make_weights(fmt, E, H, I, seed=seed, device=dev) if w is None else w
        self.x = synth.make_x(T, H, seed=seed, device=dev) if x is None else x
        self.wr = synth.make_router(E, H, seed=seed, device=dev) if wr is None else wr
        self.bias = None if bias is None else bias.to(dev)
        if isinstance(residual, torch.Tensor):
            self.residual = residual
        else:
            self.residual = synth.make_x(T, H, seed=seed + 1000, device=dev) if residual else None
        self.ow = ow

    def run(self, out=None, ws=None):
        """One moe_decode_layer_ex call (on `ws` if given, else a new zeroed
        workspace); the device status must be clean afterwards."""
        T, H, E, k = self.T, self.H, self.E, self.k
        n = binding.moe_workspace_size(self.w, T, k, self.flags)
        self.ws = binding.alloc_workspace(n) if ws is None else ws
        self.out = torch.empty((T, H), dtype=torch.bfloat16, device="cuda") if out is None else out
        self.logits = torch.empty((T, E), dtype=torch.float32, device="cuda")
        self.ids = torch.empty((T, k), dtype=torch.int32, device="cuda")
        self.gates = torch.empty((T, k), dtype=torch.float32, device="cuda")
        binding.moe_decode_layer_ex(self.x, self.wr, self.bias, self.w, k, self.out, self.ws,
                                    flags=self.flags, residual=self.residual,
                                    logits_out=self.logits, topk_ids_out=self.ids,
                                    topk_w_out=self.gates)
        torch.cuda.synchronize()
        assert binding.moe_read_status(self.ws) == 0
        return self

    # ---- oracle side
    def x_bits(self):
        if self.flags & binding.MOE_FLAG_PRENORM_RMS:
            return oracle.rmsnorm_bf16(np_(self.x), 1e-6)
        return np_(self.x)

    def check_routing(self):
        xb = self.x_bits()
        g_logits = self.logits.double().cpu().numpy()
        g_ids = self.ids.cpu().numpy()
        g_gates = self.gates.double().cpu().numpy()
        renorm = not (self.flags & binding.MOE_FLAG_NO_RENORM)
        # 1. bit-exact selection given the GPU's fp32 logits
        o_ids, o_gates = oracle.topk(g_logits, self.k, renorm)
        assert np.array_equal(o_ids, g_ids), "top-k differs on identical logits"
        assert np.abs(o_gates - g_gates).max() <= GATE_TOL
        assert np.abs(g_gates.sum(axis=1) - 1).max() <= GATE_TOL if renorm else True
        # 2. the fp32 logits are within the fp32 dot-product bound of the float64 ones
        bias = None if self.bias is None else self.bias.cpu().numpy()
        ref = oracle.router_logits(xb, np_(self.wr), bias)
        from tests import indep
        xa = np.abs(indep.bf16_to_f64(xb))
        wa = np.abs(np_(self.wr)).astype(np.float64)
        bound = 4 * self.H * 2.0 ** -24 * (xa @ wa.T) + 1e-6
        if bias is not None:
            bound += np.abs(bias) * 2.0 ** -23
        if self.flags & binding.MOE_FLAG_PRENORM_RMS:
            bound += prenorm_ambiguity(np_(self.x), self.H) @ wa.T
        assert (np.abs(g_logits - ref) <= bound).all()
        return o_ids, o_gates

    def reference(self, tokens=None):
        ids, gates = self.check_routing()
        ow = oracle_weights(self.w) if self.ow is None else self.ow
        res = None if self.residual is None else np_(self.residual)
        return oracle.moe_tokens(ow, self.x_bits(), ids, gates, tokens, res)

    def check_output(self, tokens=None, tol=REL_TOL, row_tol=None):
        """Element-by-element comparison with the oracle on the listed tokens
        (all by default).  The contract is global: max|gpu - ref| <= tol *
        max|ref| over the layer output.  Beside it the worst per-row figure,
        max_h|gpu - ref| / max_h|ref| over a token's row, is recorded for the
        session report and, with row_tol, asserted too."""
        ref = self.reference(tokens)
        got = self.out.float().cpu().numpy().astype(np.float64)
        if tokens is not None:
            got = got[np.asarray(tokens)]
        assert np.isfinite(got).all()
        err = np.abs(got - ref).max()
        scale = np.abs(ref).max()
        rows = row_errors(got, ref)
        record(self, err / scale, rows)
        assert err <= tol * scale, f"max err {err:.3e} vs {tol} * {scale:.3e}"
        if row_tol is not None:
            worst = int(np.argmax(rows))
            assert rows[worst] <= row_tol, f"row {worst}: relative error {rows[worst]:.3e}"
        return err / scale


def prenorm_ambiguity(x_bits, H):
    """Per element of bf16(RMSNorm(x)), how far the device's rounding may be
    from the oracle's.  The device computes the row scale r in fp32 (the sum of
    squares accumulated in fp32 over at most H/32 + 5 steps per value, then a
    division, a square root, a reciprocal, and the product x * r in fp32); the
    oracle computes it in float64 and rounds x * r once.  With r known to a
    relative delta, an element whose x*r*(1 - delta) and x*r*(1 + delta) round
    to different bf16 values may come out as either: the result is the gap
    between them (one ulp, or zero where the rounding is certain)."""
    from tests import indep
    xv = indep.bf16_to_f64(x_bits)
    r = 1.0 / np.sqrt((xv * xv).mean(axis=1, keepdims=True) + 1e-6)
    delta = (H / 32 + 16) * 2.0 ** -24
    lo = indep.bf16_to_f64(oracle.to_bf16_bits(xv * r * (1 - delta)))
    hi = indep.bf16_to_f64(oracle.to_bf16_bits(xv * r * (1 + delta)))
    return np.abs(hi - lo)


def row_errors(got, ref):
    """Per row: max|got - ref| / max|ref| (rows whose reference is all zero
    compare absolute errors against 1)."""
    den = np.abs(ref).max(axis=1)
    return np.abs(got - ref).max(axis=1) / np.where(den > 0, den, 1.0)


# (test, format, T, checked rows, global error, worst row error), for the
# session summary printed by conftest.py
REPORT = []


def record(case, global_err, rows):
    import os
    name = os.environ.get("PYTEST_CURRENT_TEST", "?").split(" ")[0]
    REPORT.append((name, case.fmt, case.T, len(rows), float(global_err), float(rows.max())))
