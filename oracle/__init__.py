"""CPU oracle for the HSA hot path (ctypes wrapper around hsa_oracle.c).

TEST INFRASTRUCTURE ONLY: only tests/, __graft_entry__.smoke() and bench.py's
CPU-baseline leg import this package. It never imports the CUDA library and
the CUDA library never imports it.

All arrays are numpy. Floating-point inputs are fp64 (bf16 data is widened
exactly); `f32=True` makes the chunk summaries and the selection scores follow
the fp32 definition the CUDA kernels use for the top-k decision.
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "libhsa_oracle.so")
_lib = None


def build() -> str:
    src = os.path.join(_HERE, "hsa_oracle.c")
    os.makedirs(_BUILD, exist_ok=True)
    if not (os.path.exists(_SO) and os.path.getmtime(_SO) >= os.path.getmtime(src)):
        tmp = _SO + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fopenmp", "-ffp-contract=off", "-fPIC", "-shared",
                               src, "-o", tmp, "-lm"])
        os.replace(tmp, _SO)
    return _SO


def lib():
    global _lib
    if _lib is None:
        L = ctypes.CDLL(build())
        vp, ci, cd = ctypes.c_void_p, ctypes.c_int, ctypes.c_double
        i64 = ctypes.c_int64
        L.hsa_oracle_pool.argtypes = [vp, ci, ci, ci, ci, ci, ci, vp]
        L.hsa_oracle_select.argtypes = [vp, vp, ci, ci, ci, ci, ci, ci, ci, cd, ci, vp, vp, vp, vp]
        L.hsa_oracle_forward.argtypes = [vp, vp, vp, vp, vp, ci, ci, ci, ci, ci, ci, ci, cd, ci, ci, vp, vp, vp]
        L.hsa_oracle_backward.argtypes = [vp, vp, vp, vp, vp, vp, vp, ci, ci, ci, ci, ci, ci, ci, cd, cd, ci, ci,
                                          vp, vp, vp, vp, vp, vp]
        L.hsa_oracle_select_backward.argtypes = [vp, vp, vp, vp, ci, ci, ci, ci, ci, ci, ci, cd, vp, vp, vp]
        L.hsa_oracle_decode_select.argtypes = [vp, vp, i64, ci, ci, ci, ci, ci, cd, ci, vp, vp, vp]
        L.hsa_oracle_decode_attend.argtypes = [vp, vp, vp, vp, vp, ci, ci, ci, ci, ci, ci, cd, ci, ci, vp, vp]
        for f in (L.hsa_oracle_pool, L.hsa_oracle_select, L.hsa_oracle_forward, L.hsa_oracle_backward,
                  L.hsa_oracle_select_backward,
                  L.hsa_oracle_decode_select, L.hsa_oracle_decode_attend):
            f.restype = None
        L.hsa_oracle_threads.restype = ci
        _lib = L
    return _lib


def threads() -> int:
    return int(lib().hsa_oracle_threads())


def default_scales(G: int, d: int):
    """c_sel = 1/sqrt(G*d) for the summed group query, c_att = 1/sqrt(d), as fp32 values."""
    return float(np.float32(1.0 / math.sqrt(G * d))), float(np.float32(1.0 / math.sqrt(d)))


def _f64(x):
    return np.ascontiguousarray(x, dtype=np.float64)


def _p(x):
    return ctypes.c_void_p(x.ctypes.data) if x is not None else None


def _mask(token_mask, B, L):
    if token_mask is None:
        return None
    m = np.ascontiguousarray(token_mask, dtype=np.uint8)
    assert m.shape == (B, L)
    return m


def pool(K, S, f32=False):
    """K [B, L, Hkv, d] -> K̄ [B, L//S, Hkv, d]."""
    K = _f64(K)
    B, L, Hkv, d = K.shape
    kbar = np.zeros((B, L // S, Hkv, d))
    lib().hsa_oracle_pool(_p(K), B, L, Hkv, d, S, int(f32), _p(kbar))
    return kbar


def select(q, kbar, S, topk, scale_sel=None, f32=False, token_mask=None):
    """q [B, L, Hq, d], K̄ [B, L//S, Hkv, d] -> idx [B,L,Hkv,k] int32, s_sel, gap [B,L,Hkv].

    token_mask [B, L] (optional): rows outside it are left as idx = -1, s_sel = 0, gap = 0."""
    q, kbar = _f64(q), _f64(kbar)
    B, L, Hq, d = q.shape
    Hkv = kbar.shape[2]
    if scale_sel is None:
        scale_sel = default_scales(Hq // Hkv, d)[0]
    idx = np.full((B, L, Hkv, topk), -1, dtype=np.int32)
    s_sel = np.zeros((B, L, Hkv, topk))
    gap = np.zeros((B, L, Hkv))
    m = _mask(token_mask, B, L)
    lib().hsa_oracle_select(_p(q), _p(kbar), B, L, Hq, Hkv, d, S, topk, float(scale_sel), int(f32), _p(m), _p(idx),
                            _p(s_sel), _p(gap))
    return idx, s_sel, gap


def _variant(inner, weights):
    assert inner in ("softmax", "softmax1") and weights in ("softmax", "stick")
    return int(inner == "softmax1"), int(weights == "stick")


def forward(q, K, V, idx, s_sel, S, scale_attn=None, token_mask=None, inner="softmax", weights="softmax"):
    """-> O [B, L, Hq, d], w [B, L, Hkv, k] (rows outside token_mask stay 0).

    inner: "softmax" or "softmax1" (softmax-off-by-one inside a chunk); weights:
    "softmax" or "stick" (stick-breaking chunk weights over I')."""
    q, K, V, s_sel = _f64(q), _f64(K), _f64(V), _f64(s_sel)
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    B, L, Hq, d = q.shape
    Hkv = K.shape[2]
    topk = idx.shape[-1]
    if scale_attn is None:
        scale_attn = default_scales(Hq // Hkv, d)[1]
    O = np.zeros(q.shape)  # zero pages on demand: a masked call writes only its rows
    w = np.zeros((B, L, Hkv, topk))
    m = _mask(token_mask, B, L)
    lib().hsa_oracle_forward(_p(q), _p(K), _p(V), _p(idx), _p(s_sel), B, L, Hq, Hkv, d, S, topk, float(scale_attn),
                             *_variant(inner, weights), _p(m), _p(O), _p(w))
    return O, w


def backward(q, K, V, kbar, idx, s_sel, dO, S, scale_sel=None, scale_attn=None, token_mask=None, inner="softmax",
             weights="softmax"):
    """-> dict(dq, dK, dV, dkbar, ds); with token_mask only those tokens contribute (variants as in forward)."""
    q, K, V, kbar, s_sel, dO = map(_f64, (q, K, V, kbar, s_sel, dO))
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    B, L, Hq, d = q.shape
    Hkv = K.shape[2]
    topk = idx.shape[-1]
    cs, ca = default_scales(Hq // Hkv, d)
    scale_sel = cs if scale_sel is None else scale_sel
    scale_attn = ca if scale_attn is None else scale_attn
    dq, dK, dV = np.zeros_like(q), np.zeros_like(K), np.zeros_like(V)
    dkbar = np.zeros_like(kbar)
    ds = np.zeros((B, L, Hkv, topk))
    m = _mask(token_mask, B, L)
    lib().hsa_oracle_backward(_p(q), _p(K), _p(V), _p(kbar), _p(idx), _p(s_sel), _p(dO), B, L, Hq, Hkv, d, S, topk,
                              float(scale_sel), float(scale_attn), *_variant(inner, weights), _p(m), _p(dq), _p(dK),
                              _p(dV), _p(dkbar), _p(ds))
    return dict(dq=dq, dK=dK, dV=dV, dkbar=dkbar, ds=ds)


def select_backward(q, kbar, idx, ds, S, scale_sel=None):
    """The selection chain for a given score gradient ds [B,L,Hkv,k] -> dict(dq, dK, dkbar)."""
    q, kbar, ds = _f64(q), _f64(kbar), _f64(ds)
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    B, L, Hq, d = q.shape
    Hkv = kbar.shape[2]
    topk = idx.shape[-1]
    if scale_sel is None:
        scale_sel = default_scales(Hq // Hkv, d)[0]
    dq = np.zeros_like(q)
    dK = np.zeros((B, L, Hkv, d))
    dkbar = np.zeros_like(kbar)
    lib().hsa_oracle_select_backward(_p(q), _p(kbar), _p(idx), _p(ds), B, L, Hq, Hkv, d, S, topk, float(scale_sel),
                                     _p(dq), _p(dK), _p(dkbar))
    return dict(dq=dq, dK=dK, dkbar=dkbar)


def decode_select(q, kbar, topk, scale_sel=None, f32=False):
    """q [Bq, Hq, d], K̄ [Nc, Hkv, d] -> idx, s_sel [Bq, Hkv, k], gap [Bq, Hkv]."""
    q, kbar = _f64(q), _f64(kbar)
    Bq, Hq, d = q.shape
    Nc, Hkv = kbar.shape[0], kbar.shape[1]
    if scale_sel is None:
        scale_sel = default_scales(Hq // Hkv, d)[0]
    idx = np.zeros((Bq, Hkv, topk), dtype=np.int32)
    s_sel = np.zeros((Bq, Hkv, topk))
    gap = np.zeros((Bq, Hkv))
    lib().hsa_oracle_decode_select(_p(q), _p(kbar), Nc, Bq, Hq, Hkv, d, topk, float(scale_sel), int(f32), _p(idx),
                                   _p(s_sel), _p(gap))
    return idx, s_sel, gap


def decode_attend(q, Ksel, Vsel, idx, s_sel, scale_attn=None, inner="softmax", weights="softmax"):
    """Ksel, Vsel [Bq, Hkv, k, S, d] rows of the selected chunks -> w [Bq, Hkv, k], O [Bq, Hq, d]."""
    q, Ksel, Vsel, s_sel = map(_f64, (q, Ksel, Vsel, s_sel))
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    Bq, Hq, d = q.shape
    Hkv, topk, S = Ksel.shape[1], Ksel.shape[2], Ksel.shape[3]
    if scale_attn is None:
        scale_attn = default_scales(Hq // Hkv, d)[1]
    w = np.zeros((Bq, Hkv, topk))
    O = np.zeros_like(q)
    lib().hsa_oracle_decode_attend(_p(q), _p(Ksel), _p(Vsel), _p(idx), _p(s_sel), Bq, Hq, Hkv, d, S, topk,
                                   float(scale_attn), *_variant(inner, weights), _p(w), _p(O))
    return w, O


def gather_chunks(mem, idx, S):
    """Rows of the selected chunks of a decode memory: mem [T, Hkv, d], idx [Bq, Hkv, k] -> [Bq, Hkv, k, S, d]."""
    Bq, Hkv, topk = idx.shape
    d = mem.shape[-1]
    out = np.zeros((Bq, Hkv, topk, S, d))
    for b in range(Bq):
        for g in range(Hkv):
            for j in range(topk):
                c = int(idx[b, g, j])
                if c >= 0:
                    out[b, g, j] = mem[c * S:(c + 1) * S, g, :]
    return out


def decode(q, Kmem, Vmem, kbar, S, topk, scale_sel=None, scale_attn=None, f32=False, inner="softmax",
           weights="softmax"):
    """Whole decode step for small memories (full K, V given)."""
    idx, s_sel, gap = decode_select(q, kbar, topk, scale_sel, f32)
    w, O = decode_attend(q, gather_chunks(Kmem, idx, S), gather_chunks(Vmem, idx, S), idx, s_sel, scale_attn, inner,
                         weights)
    return dict(idx=idx, s_sel=s_sel, gap=gap, w=w, O=O)
