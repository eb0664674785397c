"""Helpers that move synthetic torch inputs to numpy for the oracle."""
from types import SimpleNamespace

import numpy as np
import torch


def np_(t):
    if t is None:
        return None
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


def weights_np(w):
    return SimpleNamespace(fmt=w.fmt, E=w.E, H=w.H, I=w.I, w_gate=np_(w.w_gate),
                           w_up=np_(w.w_up), w_down=np_(w.w_down), s_gate=np_(w.s_gate),
                           s_up=np_(w.s_up), s_down=np_(w.s_down), ts_gate=np_(w.ts_gate),
                           ts_up=np_(w.ts_up), ts_down=np_(w.ts_down))


def oracle_weights(w):
    from oracle import oracle
    n = weights_np(w) if isinstance(w.w_gate, torch.Tensor) else w
    return oracle.ExpertWeights(n.fmt, n.E, n.H, n.I, n.w_gate, n.w_up, n.w_down, n.s_gate,
                                n.s_up, n.s_down, n.ts_gate, n.ts_up, n.ts_down)
