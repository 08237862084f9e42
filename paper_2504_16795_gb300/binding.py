"""Thin ctypes binding of libhsa.so (the C ABI declared in include/hsa.h).

Argument marshalling only: every computation runs in the CUDA library. Torch
tensors supply device memory and the current stream. If the library is not
built the first call raises; there is no fallback path.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from typing import Optional

import torch

from . import build as _build

HSA_OP_SELECT, HSA_OP_INDEX, HSA_OP_FORWARD, HSA_OP_BACKWARD = 1, 2, 3, 4
HSA_OP_BACKWARD_ATTENTION, HSA_OP_SELECT_BACKWARD = 5, 6
CHUNK = 64


class HsaError(RuntimeError):
    def __init__(self, status: int, what: str):
        super().__init__(f"{what}: {status_string(status)}")
        self.status = status


class _Shape(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("L", ctypes.c_int), ("Hq", ctypes.c_int), ("Hkv", ctypes.c_int),
                ("d", ctypes.c_int), ("S", ctypes.c_int), ("topk", ctypes.c_int),
                ("scale_sel", ctypes.c_float), ("scale_attn", ctypes.c_float), ("flags", ctypes.c_int)]


class _DecodeShape(ctypes.Structure):
    _fields_ = [("Bq", ctypes.c_int), ("Hq", ctypes.c_int), ("Hkv", ctypes.c_int), ("d", ctypes.c_int),
                ("S", ctypes.c_int), ("topk", ctypes.c_int), ("n_chunks", ctypes.c_longlong),
                ("scale_sel", ctypes.c_float), ("scale_attn", ctypes.c_float), ("flags", ctypes.c_int),
                ("capacity_chunks", ctypes.c_longlong)]


def _flags(inner: str, weights: str) -> int:
    if inner not in ("softmax", "softmax1") or weights not in ("softmax", "stick"):
        raise ValueError(f"unknown variant: inner={inner!r}, weights={weights!r}")
    return (1 if inner == "softmax1" else 0) | (2 if weights == "stick" else 0)


@dataclass(frozen=True)
class Shape:
    """Prefill problem: q [B, L, Hq, d], K, V [B, L, Hkv, d], chunk S, top-k."""
    B: int
    L: int
    Hq: int
    Hkv: int
    d: int
    S: int = CHUNK
    topk: int = 8
    scale_sel: float = 0.0   # <= 0: 1/sqrt(G*d)
    scale_attn: float = 0.0  # <= 0: 1/sqrt(d)
    inner: str = "softmax"    # or "softmax1": softmax-off-by-one inside a chunk
    weights: str = "softmax"  # or "stick": stick-breaking chunk weights

    @property
    def flags(self) -> int:
        return _flags(self.inner, self.weights)

    @property
    def G(self) -> int:
        return self.Hq // self.Hkv

    @property
    def Nc(self) -> int:
        return self.L // self.S

    def c(self) -> _Shape:
        return _Shape(self.B, self.L, self.Hq, self.Hkv, self.d, self.S, self.topk, self.scale_sel, self.scale_attn,
                      self.flags)


@dataclass(frozen=True)
class DecodeShape:
    Bq: int
    Hq: int
    Hkv: int
    d: int
    n_chunks: int
    S: int = CHUNK
    topk: int = 8
    scale_sel: float = 0.0
    scale_attn: float = 0.0
    inner: str = "softmax"
    weights: str = "softmax"
    capacity_chunks: int = 0  # a growing memory's capacity (0: n_chunks)

    def c(self) -> _DecodeShape:
        return _DecodeShape(self.Bq, self.Hq, self.Hkv, self.d, self.S, self.topk, self.n_chunks, self.scale_sel,
                            self.scale_attn, _flags(self.inner, self.weights), self.capacity_chunks)


_lib = None


def lib_path() -> str:
    return _build.LIB


def load():
    """Load libhsa.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_build.LIB):
        raise RuntimeError(f"HSA CUDA library not built ({_build.LIB}); run paper_2504_16795_gb300.build.build()")
    L = ctypes.CDLL(_build.LIB)
    vp, sz, i = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int
    sp = ctypes.POINTER(_Shape)
    dp = ctypes.POINTER(_DecodeShape)
    L.hsa_status_string.restype = ctypes.c_char_p
    L.hsa_status_string.argtypes = [i]
    L.hsa_version.restype = i
    L.hsa_kernel_launches.restype = ctypes.c_ulonglong
    L.hsa_kernel_launches.argtypes = []
    L.hsa_status_bytes.restype = sz
    L.hsa_status_bytes.argtypes = []
    L.hsa_check.restype = i
    L.hsa_check.argtypes = [vp, sz, vp]
    L.hsa_selftest_wait_timeout.restype = i
    L.hsa_selftest_wait_timeout.argtypes = [ctypes.c_ulonglong, vp, sz, vp]
    L.hsa_selftest_score_tile.restype = i
    L.hsa_selftest_score_tile.argtypes = [i, vp, vp, vp, vp, sz, vp]
    L.hsa_workspace_size.restype = sz
    L.hsa_workspace_size.argtypes = [i, sp]
    L.hsa_decode_workspace_size.restype = sz
    L.hsa_decode_workspace_size.argtypes = [dp]
    L.hsa_chunk_pool.argtypes = [sp, vp, vp, vp, vp]
    L.hsa_select_topk.argtypes = [sp, vp, vp, vp, vp, vp, sz, vp]
    L.hsa_build_index.argtypes = [sp, vp, vp, vp, vp, sz, vp]
    L.hsa_forward.argtypes = [sp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
    L.hsa_backward.argtypes = [sp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
    L.hsa_backward_attention.argtypes = [sp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
    L.hsa_select_backward.argtypes = [sp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
    L.hsa_decode.argtypes = [dp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
    L.hsa_decode_noalloc.argtypes = [dp, vp, vp, vp, vp, vp, vp, vp, vp, vp]
    L.hsa_decode_index_size.restype = sz
    L.hsa_decode_index_size.argtypes = [dp]
    L.hsa_decode_index.argtypes = [dp, vp, vp, sz, vp]
    L.hsa_decode_indexed_workspace_size.restype = sz
    L.hsa_decode_indexed_workspace_size.argtypes = [dp]
    L.hsa_decode_indexed.argtypes = [dp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
    L.hsa_memory_append.argtypes = [dp, ctypes.c_longlong, ctypes.c_longlong, vp, vp, vp, vp, vp, vp, sz, vp]
    for f in (L.hsa_chunk_pool, L.hsa_select_topk, L.hsa_build_index, L.hsa_forward, L.hsa_backward,
              L.hsa_decode, L.hsa_decode_noalloc, L.hsa_decode_index, L.hsa_decode_indexed, L.hsa_memory_append):
        f.restype = i
    _lib = L
    return L


def kernel_launches() -> int:
    """Kernels launched by libhsa.so since it was loaded."""
    return int(load().hsa_kernel_launches())


def status_bytes() -> int:
    """Bytes of the status header that starts every workspace."""
    return int(load().hsa_status_bytes())


def check(ws: Optional[torch.Tensor]) -> None:
    """hsa_check: wait for the current stream of ws's device and raise HsaError if a bounded wait gave up in a
    call that used this workspace since its last check (the status word is cleared). None: nothing to check."""
    if ws is None:
        return
    _check(load().hsa_check(_ptr(ws), ws.numel() * ws.element_size(), _stream(ws.device)), "hsa_check")


def selftest_wait_timeout(limit_ns: int, ws: torch.Tensor) -> None:
    """Launch the bounded-wait self-test (a wait nothing completes, given up after limit_ns); it sets the
    status word of workspace ws, which the next check(ws) reports."""
    _check(load().hsa_selftest_wait_timeout(int(limit_ns), _ptr(ws), ws.numel() * ws.element_size(),
                                            _stream(ws.device)), "hsa_selftest_wait_timeout")


def selftest_score_tile(A: torch.Tensor, B: torch.Tensor, ws: Optional[torch.Tensor] = None) -> torch.Tensor:
    """hsa_selftest_score_tile: A [128, d] and B [64, d] bf16 -> C [128, 64] fp32 from the selection's
    tensor-core score pass (for measuring its accumulation rounding)."""
    d = int(A.shape[1])
    _need(A, "A", torch.bfloat16, (128, d))
    _need(B, "B", torch.bfloat16, (64, d))
    C = torch.empty((128, 64), dtype=torch.float32, device=A.device)
    ws = ws if ws is not None else new_workspace(status_bytes(), A.device)
    _check(load().hsa_selftest_score_tile(d, _ptr(A), _ptr(B), _ptr(C), _ptr(ws), ws.numel(), _stream(A.device)),
           "hsa_selftest_score_tile")
    return C


def status_string(status: int) -> str:
    return load().hsa_status_string(int(status)).decode()


def _ptr(t: Optional[torch.Tensor]):
    return ctypes.c_void_p(t.data_ptr()) if t is not None else ctypes.c_void_p(0)


def _stream(device) -> ctypes.c_void_p:
    return ctypes.c_void_p(torch.cuda.current_stream(device).cuda_stream)


def _check(rc: int, what: str):
    if rc != 0:
        raise HsaError(rc, what)


def _need(t: torch.Tensor, name: str, dtype, shape):
    if t.dtype != dtype:
        raise TypeError(f"{name}: expected {dtype}, got {t.dtype}")
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name}: expected shape {tuple(shape)}, got {tuple(t.shape)}")
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError(f"{name}: must be a contiguous CUDA tensor")


def workspace_size(op: int, shape: Shape) -> int:
    s = shape.c()
    return int(load().hsa_workspace_size(op, ctypes.byref(s)))


def decode_workspace_size(shape: DecodeShape) -> int:
    s = shape.c()
    return int(load().hsa_decode_workspace_size(ctypes.byref(s)))


def new_workspace(nbytes: int, device) -> Optional[torch.Tensor]:
    """A caller-owned workspace of nbytes (None for 0) with its status header cleared."""
    if nbytes == 0:
        return None
    ws = torch.empty(nbytes, dtype=torch.uint8, device=device)
    ws[:min(nbytes, status_bytes())].zero_()
    return ws


def _workspace(nbytes: int, device, ws: Optional[torch.Tensor]):
    if nbytes == 0:
        return None
    if ws is not None and ws.numel() * ws.element_size() >= nbytes:
        return ws
    return new_workspace(nbytes, device)


def chunk_pool(shape: Shape, K: torch.Tensor, kbar32=None, kbar16=None, want_bf16: bool = True):
    """K̄ (fp32, and its bf16 rounding) of every complete chunk."""
    _need(K, "K", torch.bfloat16, (shape.B, shape.L, shape.Hkv, shape.d))
    dev = K.device
    if kbar32 is None:
        kbar32 = torch.empty((shape.B, shape.Nc, shape.Hkv, shape.d), dtype=torch.float32, device=dev)
    if kbar16 is None and want_bf16:
        kbar16 = torch.empty((shape.B, shape.Nc, shape.Hkv, shape.d), dtype=torch.bfloat16, device=dev)
    s = shape.c()
    _check(load().hsa_chunk_pool(ctypes.byref(s), _ptr(K), _ptr(kbar32), _ptr(kbar16), _stream(dev)),
           "hsa_chunk_pool")
    return kbar32, kbar16


def select_topk(shape: Shape, q: torch.Tensor, kbar32: torch.Tensor, idx=None, s_sel=None, ws=None):
    _need(q, "q", torch.bfloat16, (shape.B, shape.L, shape.Hq, shape.d))
    _need(kbar32, "kbar32", torch.float32, (shape.B, shape.Nc, shape.Hkv, shape.d))
    dev = q.device
    out_shape = (shape.B, shape.L, shape.Hkv, shape.topk)
    idx = torch.empty(out_shape, dtype=torch.int32, device=dev) if idx is None else idx
    s_sel = torch.empty(out_shape, dtype=torch.float32, device=dev) if s_sel is None else s_sel
    nb = workspace_size(HSA_OP_SELECT, shape)
    w = _workspace(nb, dev, ws)
    s = shape.c()
    _check(load().hsa_select_topk(ctypes.byref(s), _ptr(q), _ptr(kbar32), _ptr(idx), _ptr(s_sel), _ptr(w), nb,
                                  _stream(dev)), "hsa_select_topk")
    return idx, s_sel


def build_index(shape: Shape, idx: torch.Tensor, offsets=None, entries=None, ws=None):
    _need(idx, "idx", torch.int32, (shape.B, shape.L, shape.Hkv, shape.topk))
    dev = idx.device
    nkeys = shape.B * shape.Hkv * shape.Nc
    offsets = torch.empty(nkeys + 1, dtype=torch.int32, device=dev) if offsets is None else offsets
    entries = torch.empty(max(1, idx.numel()), dtype=torch.int32, device=dev) if entries is None else entries
    nb = workspace_size(HSA_OP_INDEX, shape)
    w = _workspace(nb, dev, ws)
    s = shape.c()
    _check(load().hsa_build_index(ctypes.byref(s), _ptr(idx), _ptr(offsets), _ptr(entries), _ptr(w), nb,
                                  _stream(dev)), "hsa_build_index")
    return offsets, entries


def forward(shape: Shape, q, K, V, idx, s_sel, offsets, entries, O=None, w=None, ws=None):
    _need(q, "q", torch.bfloat16, (shape.B, shape.L, shape.Hq, shape.d))
    _need(K, "K", torch.bfloat16, (shape.B, shape.L, shape.Hkv, shape.d))
    _need(V, "V", torch.bfloat16, (shape.B, shape.L, shape.Hkv, shape.d))
    _need(idx, "idx", torch.int32, (shape.B, shape.L, shape.Hkv, shape.topk))
    _need(s_sel, "s_sel", torch.float32, (shape.B, shape.L, shape.Hkv, shape.topk))
    dev = q.device
    O = torch.empty_like(q) if O is None else O
    w = torch.empty_like(s_sel) if w is None else w
    nb = workspace_size(HSA_OP_FORWARD, shape)
    wsp = _workspace(nb, dev, ws)
    s = shape.c()
    _check(load().hsa_forward(ctypes.byref(s), _ptr(q), _ptr(K), _ptr(V), _ptr(idx), _ptr(s_sel), _ptr(offsets),
                              _ptr(entries), _ptr(O), _ptr(w), _ptr(wsp), nb, _stream(dev)), "hsa_forward")
    return O, w


def backward(shape: Shape, q, K, V, kbar32, idx, w, O, dO, offsets, entries, dq=None, dK=None, dV=None, ws=None):
    _need(dO, "dO", torch.bfloat16, (shape.B, shape.L, shape.Hq, shape.d))
    _need(O, "O", torch.bfloat16, (shape.B, shape.L, shape.Hq, shape.d))
    dev = q.device
    dq = torch.empty(q.shape, dtype=torch.float32, device=dev) if dq is None else dq
    dK = torch.empty(K.shape, dtype=torch.float32, device=dev) if dK is None else dK
    dV = torch.empty(V.shape, dtype=torch.float32, device=dev) if dV is None else dV
    nb = workspace_size(HSA_OP_BACKWARD, shape)
    wsp = _workspace(nb, dev, ws)
    s = shape.c()
    _check(load().hsa_backward(ctypes.byref(s), _ptr(q), _ptr(K), _ptr(V), _ptr(kbar32), _ptr(idx), _ptr(w), _ptr(O),
                               _ptr(dO), _ptr(offsets), _ptr(entries), _ptr(dq), _ptr(dK), _ptr(dV), _ptr(wsp), nb,
                               _stream(dev)), "hsa_backward")
    return dq, dK, dV


def backward_attention(shape: Shape, q, K, V, idx, w, dO, offsets, entries, ds_accum=None, dq=None, dK=None, dV=None,
                       ws=None):
    """The attention's gradients of one layer; its score gradient is added into ds_accum (zeros if None)."""
    _need(dO, "dO", torch.bfloat16, (shape.B, shape.L, shape.Hq, shape.d))
    dev = q.device
    dq = torch.empty(q.shape, dtype=torch.float32, device=dev) if dq is None else dq
    dK = torch.empty(K.shape, dtype=torch.float32, device=dev) if dK is None else dK
    dV = torch.empty(V.shape, dtype=torch.float32, device=dev) if dV is None else dV
    if ds_accum is None:
        ds_accum = torch.zeros((shape.B, shape.L, shape.Hkv, shape.topk), dtype=torch.float32, device=dev)
    nb = workspace_size(HSA_OP_BACKWARD_ATTENTION, shape)
    wsp = _workspace(nb, dev, ws)
    s = shape.c()
    _check(load().hsa_backward_attention(ctypes.byref(s), _ptr(q), _ptr(K), _ptr(V), _ptr(idx), _ptr(w), _ptr(dO),
                                         _ptr(offsets), _ptr(entries), _ptr(dq), _ptr(dK), _ptr(dV), _ptr(ds_accum),
                                         _ptr(wsp), nb, _stream(dev)), "hsa_backward_attention")
    return dq, dK, dV, ds_accum


def select_backward(shape: Shape, q_sel, kbar_sel, idx, ds, offsets, entries, dq_sel=None, dK_sel=None, ws=None):
    """The selection chain once for the summed score gradient: (dq_sel, dK_sel)."""
    _need(q_sel, "q_sel", torch.bfloat16, (shape.B, shape.L, shape.Hq, shape.d))
    dev = q_sel.device
    dq_sel = torch.empty(q_sel.shape, dtype=torch.float32, device=dev) if dq_sel is None else dq_sel
    if dK_sel is None:
        dK_sel = torch.empty((shape.B, shape.L, shape.Hkv, shape.d), dtype=torch.float32, device=dev)
    nb = workspace_size(HSA_OP_SELECT_BACKWARD, shape)
    wsp = _workspace(nb, dev, ws)
    s = shape.c()
    _check(load().hsa_select_backward(ctypes.byref(s), _ptr(q_sel), _ptr(kbar_sel), _ptr(idx), _ptr(ds), _ptr(offsets),
                                      _ptr(entries), _ptr(dq_sel), _ptr(dK_sel), _ptr(wsp), nb, _stream(dev)),
           "hsa_select_backward")
    return dq_sel, dK_sel


def decode(shape: DecodeShape, q, K_mem, V_mem, kbar32, O=None, idx=None, s_sel=None, w=None, ws=None):
    """hsa_decode. K_mem and V_mem may be CUDA tensors or pinned host tensors (read over the CPU-GPU
    link); q, kbar32 and the outputs live on the device."""
    _need(q, "q", torch.bfloat16, (shape.Bq, shape.Hq, shape.d))
    dev = q.device
    O = torch.empty_like(q) if O is None else O
    out = (shape.Bq, shape.Hkv, shape.topk)
    idx = torch.empty(out, dtype=torch.int32, device=dev) if idx is None else idx
    s_sel = torch.empty(out, dtype=torch.float32, device=dev) if s_sel is None else s_sel
    w = torch.empty(out, dtype=torch.float32, device=dev) if w is None else w
    nb = decode_workspace_size(shape)
    wsp = _workspace(nb, dev, ws)
    s = shape.c()
    _check(load().hsa_decode(ctypes.byref(s), _ptr(q), _ptr(K_mem), _ptr(V_mem), _ptr(kbar32), _ptr(O), _ptr(idx),
                             _ptr(s_sel), _ptr(w), _ptr(wsp), nb, _stream(dev)), "hsa_decode")
    return O, idx, s_sel, w


def decode_noalloc(shape: DecodeShape, q, K_mem, V_mem, kbar32, O, idx, s_sel, w):
    """hsa_decode_noalloc: decode into caller-provided outputs, scratch owned by the library.

    Calls on one device share the library's scratch; callers serialise them."""
    _need(q, "q", torch.bfloat16, (shape.Bq, shape.Hq, shape.d))
    _need(O, "O", torch.bfloat16, (shape.Bq, shape.Hq, shape.d))
    out = (shape.Bq, shape.Hkv, shape.topk)
    _need(idx, "idx", torch.int32, out)
    _need(s_sel, "s_sel", torch.float32, out)
    _need(w, "w", torch.float32, out)
    s = shape.c()
    with torch.cuda.device(q.device):  # the library looks up its scratch on the current device
        _check(load().hsa_decode_noalloc(ctypes.byref(s), _ptr(q), _ptr(K_mem), _ptr(V_mem), _ptr(kbar32), _ptr(O),
                                         _ptr(idx), _ptr(s_sel), _ptr(w), _stream(q.device)), "hsa_decode_noalloc")
    return O, idx, s_sel, w


def decode_index(shape: DecodeShape, kbar32, index=None):
    """The memory index of hsa_decode_indexed (built once per memory); None when not needed."""
    s = shape.c()
    nb = int(load().hsa_decode_index_size(ctypes.byref(s)))
    if nb == 0:
        return None
    dev = kbar32.device
    index = torch.empty(nb, dtype=torch.uint8, device=dev) if index is None else index
    _check(load().hsa_decode_index(ctypes.byref(s), _ptr(kbar32), _ptr(index), nb, _stream(dev)), "hsa_decode_index")
    return index


def decode_indexed(shape: DecodeShape, q, K_mem, V_mem, kbar32, index, O=None, idx=None, s_sel=None, w=None,
                   ws=None):
    """hsa_decode_indexed: as decode, scanning the memory index (decode_index) on the tensor cores."""
    _need(q, "q", torch.bfloat16, (shape.Bq, shape.Hq, shape.d))
    dev = q.device
    O = torch.empty_like(q) if O is None else O
    out = (shape.Bq, shape.Hkv, shape.topk)
    idx = torch.empty(out, dtype=torch.int32, device=dev) if idx is None else idx
    s_sel = torch.empty(out, dtype=torch.float32, device=dev) if s_sel is None else s_sel
    w = torch.empty(out, dtype=torch.float32, device=dev) if w is None else w
    s = shape.c()
    nb = int(load().hsa_decode_indexed_workspace_size(ctypes.byref(s)))
    wsp = _workspace(nb, dev, ws)
    _check(load().hsa_decode_indexed(ctypes.byref(s), _ptr(q), _ptr(K_mem), _ptr(V_mem), _ptr(kbar32), _ptr(index),
                                     _ptr(O), _ptr(idx), _ptr(s_sel), _ptr(w), _ptr(wsp), nb, _stream(dev)),
           "hsa_decode_indexed")
    return O, idx, s_sel, w


def memory_append(shape: DecodeShape, n_tokens: int, K_new, V_new, K_mem, V_mem, kbar32, index=None) -> int:
    """hsa_memory_append: append K_new, V_new [n_new, Hkv, d] to a memory holding n_tokens tokens (rows
    stored, completed chunks pooled into kbar32 and entered in index); returns the new token count.

    K_new, V_new, K_mem, V_mem may be CUDA tensors or pinned host tensors; kbar32 and index live on the device."""
    n_new = int(K_new.shape[0])
    for t, name in ((K_new, "K_new"), (V_new, "V_new")):
        if t.dtype != torch.bfloat16 or tuple(t.shape) != (n_new, shape.Hkv, shape.d) or not t.is_contiguous():
            raise ValueError(f"{name}: expected a contiguous bf16 tensor of shape {(n_new, shape.Hkv, shape.d)}")
    nb = index.numel() * index.element_size() if index is not None else 0
    s = shape.c()
    _check(load().hsa_memory_append(ctypes.byref(s), int(n_tokens), n_new, _ptr(K_new), _ptr(V_new), _ptr(K_mem),
                                    _ptr(V_mem), _ptr(kbar32), _ptr(index), nb, _stream(kbar32.device)),
           "hsa_memory_append")
    return int(n_tokens) + n_new


class Workspaces:
    """Caller-owned scratch for a fixed shape, reused across calls (allocated by torch)."""

    def __init__(self, shape: Shape, device):
        self.shape = shape
        self.select = _workspace(workspace_size(HSA_OP_SELECT, shape), device, None)
        self.index = _workspace(workspace_size(HSA_OP_INDEX, shape), device, None)
        self.forward = _workspace(workspace_size(HSA_OP_FORWARD, shape), device, None)
        self.backward = _workspace(workspace_size(HSA_OP_BACKWARD, shape), device, None)

    def check(self) -> None:
        """check() every workspace of the set."""
        for ws in (self.select, self.index, self.forward, self.backward):
            check(ws)


def hsa_forward_path(shape: Shape, q, K, V, wss: Optional[Workspaces] = None):
    """pool -> select -> inverse index -> attention + merge. Returns a dict of every intermediate."""
    wss = wss or Workspaces(shape, q.device)
    kbar32, kbar16 = chunk_pool(shape, K)
    idx, s_sel = select_topk(shape, q, kbar32, ws=wss.select)
    offsets, entries = build_index(shape, idx, ws=wss.index)
    O, w = forward(shape, q, K, V, idx, s_sel, offsets, entries, ws=wss.forward)
    return dict(kbar32=kbar32, kbar16=kbar16, idx=idx, s_sel=s_sel, offsets=offsets, entries=entries, O=O, w=w)


def hsa_backward_path(shape: Shape, q, K, V, fwd: dict, dO, wss: Optional[Workspaces] = None):
    wss = wss or Workspaces(shape, q.device)
    return backward(shape, q, K, V, fwd["kbar32"], fwd["idx"], fwd["w"], fwd["O"], dO, fwd["offsets"],
                    fwd["entries"], ws=wss.backward)
