"""Shared helpers for the GPU parity tests: seeded inputs for both sides, the
oracle run, and the comparison bars.

Bars (fixed by the operator's parity contract):
  * chunk summaries and selection: bit-exact (both sides take the fp32
    decision with the same operation order); rows whose oracle k-th and
    (k+1)-th scores differ by < 1e-4 are counted and reported;
  * outputs and gradients: max-abs <= 2e-2 and relative RMS <= 1e-2 against
    the fp64 oracle.
"""
from __future__ import annotations

import numpy as np

import oracle
import synth

MAX_ABS = 2e-2
REL_RMS = 1e-2
TIE_WINDOW = 1e-4


def to_device_bf16(bits: np.ndarray, device="cuda"):
    import torch

    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(device)


def bf16_tensor_to_f64(t) -> np.ndarray:
    import torch

    return synth.bf16_to_f64(t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16))


def rel_rms(got, want) -> float:
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    den = np.sqrt(np.mean(want ** 2))
    return float(np.sqrt(np.mean((got - want) ** 2)) / (den if den > 0 else 1.0))


def assert_close(name, got, want, max_abs=MAX_ABS, rel=REL_RMS):
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    assert got.shape == want.shape, (name, got.shape, want.shape)
    assert np.isfinite(got).all(), f"{name}: non-finite values"
    err = np.abs(got - want).max() if got.size else 0.0
    rr = rel_rms(got, want) if got.size else 0.0
    assert err <= max_abs, f"{name}: max-abs {err:.3e} > {max_abs}"
    assert rr <= rel, f"{name}: rel-RMS {rr:.3e} > {rel}"
    return err, rr


def host_inputs(w: synth.Workload, with_dO=True):
    """bf16 bit patterns of q, K, V (and dO) for the whole workload."""
    out = {}
    for name in ("q", "K", "V") + (("dO",) if with_dO else ()):
        dims = w.dims(name)
        out[name] = synth.host_tensor(w, name, (0, 0, 0, 0), dims)
    return out


def oracle_prefill(w: synth.Workload, bits: dict, backward=True, token_mask=None, inner="softmax", weights="softmax"):
    """Oracle results for a prefill workload from its bf16 inputs (variants as in oracle.forward)."""
    q = synth.bf16_to_f64(bits["q"])
    K = synth.bf16_to_f64(bits["K"])
    V = synth.bf16_to_f64(bits["V"])
    S, k = w.S, w.topk
    kbar32 = oracle.pool(K, S, f32=True)
    idx, s_sel, gap = oracle.select(q, kbar32, S, k, f32=True, token_mask=token_mask)
    O, wts = oracle.forward(q, K, V, idx, s_sel, S, token_mask=token_mask, inner=inner, weights=weights)
    res = dict(kbar32=kbar32, idx=idx, s_sel=s_sel, gap=gap, O=O, w=wts)
    if backward:
        dO = synth.bf16_to_f64(bits["dO"])
        kbar64 = oracle.pool(K, S)
        res.update(oracle.backward(q, K, V, kbar64, idx, s_sel, dO, S, token_mask=token_mask, inner=inner,
                                   weights=weights))
    return res
