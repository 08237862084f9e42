"""Seeded synthetic inputs for the HSA workloads (test and benchmark infrastructure).

The paper trains on text corpora (Pile, PG19, ...) and evaluates passkey and
RULER retrieval; none of that data is used here. These seeded tensors stand in
for those workloads in shape only: bf16 q, K, V, dO drawn i.i.d. from an
(Irwin-Hall(12)) standard normal, plus the additive structure each workload
defines (per-chunk key offsets, planted "needle" chunks aligned with some
queries).

Every element is a pure function of (seed, flat index), so the CPU oracle can
draw any slice on its own while the CUDA path fills whole tensors on the
device; `synth_host.c` and `synth_dev.cu` implement the same definition
independently and a test checks them bit for bit. This module holds no
arithmetic of the attention method.
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
from dataclasses import dataclass
from typing import Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_HOST_SO = os.path.join(_BUILD, "libsynth_host.so")
_DEV_SO = os.path.join(_BUILD, "libsynth_dev.so")

_host_lib = None
_dev_lib = None


def _newer(target: str, sources: Sequence[str]) -> bool:
    if not os.path.exists(target):
        return False
    t = os.path.getmtime(target)
    return all(os.path.getmtime(s) <= t for s in sources)


def build_host() -> str:
    os.makedirs(_BUILD, exist_ok=True)
    src = os.path.join(_HERE, "synth_host.c")
    if not _newer(_HOST_SO, [src]):
        tmp = _HOST_SO + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fopenmp", "-ffp-contract=off", "-fPIC",
                               "-shared", src, "-o", tmp])
        os.replace(tmp, _HOST_SO)
    return _HOST_SO


def build_device() -> str:
    os.makedirs(_BUILD, exist_ok=True)
    src = os.path.join(_HERE, "synth_dev.cu")
    hdr = os.path.join(_HERE, "synth.h")
    if not _newer(_DEV_SO, [src, hdr]):
        tmp = _DEV_SO + f".tmp{os.getpid()}"
        subprocess.check_call(["nvcc", "-O3", "-std=c++17", "-gencode", "arch=compute_103a,code=sm_103a",
                               "-lineinfo", "-Xcompiler", "-fPIC", "-shared", "-I", _HERE, src, "-o", tmp])
        os.replace(tmp, _DEV_SO)
    return _DEV_SO


def host_lib():
    global _host_lib
    if _host_lib is None:
        lib = ctypes.CDLL(build_host())
        i64p = ctypes.POINTER(ctypes.c_int64)
        lib.synth_box_f32.argtypes = [ctypes.c_uint64, i64p, i64p, i64p, ctypes.c_void_p]
        lib.synth_box_bf16.argtypes = [ctypes.c_uint64, i64p, i64p, i64p, ctypes.c_void_p]
        lib.synth_draws.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int64, ctypes.c_void_p]
        lib.synth_draws_state.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int64, ctypes.c_void_p]
        lib.synth_add_f32_to_bf16.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64]
        lib.synth_bf16_to_f64.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64]
        _host_lib = lib
    return _host_lib


def dev_lib():
    global _dev_lib
    if _dev_lib is None:
        lib = ctypes.CDLL(build_device())
        lib.synth_dev_fill_bf16.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_uint64, ctypes.c_int64,
                                            ctypes.c_void_p]
        lib.synth_dev_add_rows.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p,
                                           ctypes.c_int64, ctypes.c_int64, ctypes.c_void_p]
        lib.synth_dev_add_chunk_offsets.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                                    ctypes.c_int, ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p]
        for f in (lib.synth_dev_fill_bf16, lib.synth_dev_add_rows, lib.synth_dev_add_chunk_offsets):
            f.restype = ctypes.c_int
        _dev_lib = lib
    return _dev_lib


def _arr4(v):
    a = (ctypes.c_int64 * 4)(*[int(x) for x in v])
    return a


# --------------------------------------------------------------------------- raw draws

def draws(seed: int, n0: int, count: int) -> np.ndarray:
    out = np.empty(count, dtype=np.uint64)
    host_lib().synth_draws(ctypes.c_uint64(seed), ctypes.c_uint64(n0), count, out.ctypes.data)
    return out


def draws_from_state(s0: int, n0: int, count: int) -> np.ndarray:
    out = np.empty(count, dtype=np.uint64)
    host_lib().synth_draws_state(ctypes.c_uint64(s0), ctypes.c_uint64(n0), count, out.ctypes.data)
    return out


def box(seed: int, dims: Sequence[int], lo: Sequence[int], hi: Sequence[int], dtype: str = "bf16") -> np.ndarray:
    """The box lo <= i < hi of the 4-D tensor whose flat element f is ih12(seed, f)."""
    dims = list(dims) + [1] * (4 - len(dims))
    lo = list(lo) + [0] * (4 - len(lo))
    hi = list(hi) + [1] * (4 - len(hi))
    shape = [max(0, h - l) for l, h in zip(lo, hi)]
    if dtype == "bf16":
        out = np.zeros(shape, dtype=np.uint16)
        fn = host_lib().synth_box_bf16
    else:
        out = np.zeros(shape, dtype=np.float32)
        fn = host_lib().synth_box_f32
    if out.size:
        fn(ctypes.c_uint64(seed), _arr4(dims), _arr4(lo), _arr4(hi), out.ctypes.data)
    return out


def bf16_to_f32(x: np.ndarray) -> np.ndarray:
    return (x.astype(np.uint32) << np.uint32(16)).view(np.float32)


def bf16_to_f64(x: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to fp64."""
    x = np.ascontiguousarray(x, dtype=np.uint16)
    out = np.empty(x.shape, dtype=np.float64)
    if x.size:
        host_lib().synth_bf16_to_f64(x.ctypes.data, out.ctypes.data, x.size)
    return out


def f32_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even of finite fp32 values to bf16 bit patterns."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))
    return (u >> np.uint64(16)).astype(np.uint16)


def add_to_bf16(x: np.ndarray, add: np.ndarray) -> np.ndarray:
    """bf16(float(x) + add) with one fp32 addition per element."""
    return f32_to_bf16(bf16_to_f32(x) + np.asarray(add, dtype=np.float32))


# --------------------------------------------------------------------------- workloads

@dataclass(frozen=True)
class Workload:
    """One synthetic HSA workload; shapes follow the paper's operator statement."""
    name: str
    number: int
    B: int
    L: int
    S: int
    Hq: int
    Hkv: int
    d: int
    topk: int
    backward: bool = True
    decode: bool = False
    chunk_offset_sigma: float = 0.0  # K += N(0, sigma^2) drawn once per (b, chunk, g)
    needle_chunks: int = 0           # prefill: planted chunks aligned with needle queries
    needle_query_every: int = 0      # prefill: a token carries the needle if draw % every == 0
    needle_norm: float = 3.0
    Bq: int = 0                      # decode: number of query tokens

    @property
    def G(self) -> int:
        return self.Hq // self.Hkv

    @property
    def Nc(self) -> int:
        return self.L // self.S

    def seed(self, tensor: str) -> int:
        base = {"q": 1000, "K": 2000, "V": 3000, "dO": 4000, "needle": 5000, "offset": 6000}[tensor]
        return base + self.number

    def dims(self, tensor: str):
        if self.decode:
            if tensor == "q":
                return (1, self.Bq, self.Hq, self.d)
            return (1, self.L, self.Hkv, self.d)
        if tensor in ("q", "dO"):
            return (self.B, self.L, self.Hq, self.d)
        return (self.B, self.L, self.Hkv, self.d)

    def with_(self, **kw) -> "Workload":
        d = dict(self.__dict__)
        d.update(kw)
        return Workload(**d)


WORKLOADS = {
    1: Workload("tiny", 1, B=1, L=1024, S=64, Hq=4, Hkv=1, d=64, topk=4),
    2: Workload("pretrain-4k", 2, B=8, L=4096, S=64, Hq=16, Hkv=2, d=128, topk=8, chunk_offset_sigma=0.5),
    3: Workload("long-32k", 3, B=2, L=32768, S=64, Hq=32, Hkv=4, d=128, topk=8),
    4: Workload("prefill-1m", 4, B=1, L=1 << 20, S=64, Hq=16, Hkv=1, d=128, topk=16, backward=False,
                needle_chunks=32, needle_query_every=8),
    5: Workload("decode-64m", 5, B=1, L=1 << 26, S=64, Hq=8, Hkv=1, d=128, topk=8, backward=False, decode=True,
                Bq=64, needle_chunks=64),
}


def needle_direction(w: Workload, which: int = 0) -> np.ndarray:
    """A unit direction drawn from the needle stream, scaled to norm w.needle_norm (fp32)."""
    raw = box(w.seed("needle"), (1 << 20, 1, 1, w.d), (which, 0, 0, 0), (which + 1, 1, 1, w.d), "f32")
    v = raw.reshape(-1).astype(np.float64)
    v = v / math.sqrt(float(np.dot(v, v))) * w.needle_norm
    return v.astype(np.float32)


def needle_chunk_ids(w: Workload) -> np.ndarray:
    """Distinct planted chunks: prefill draws from [1, Nc), decode from [0, Nc) (one per query)."""
    lo = 0 if w.decode else 1
    span = w.Nc - lo
    want = min(w.needle_chunks, span)
    chosen, seen, n = [], set(), 0
    while len(chosen) < want:
        r = int(draws(w.seed("needle") + 77, n, 1)[0])
        n += 1
        c = lo + r % span
        if c not in seen:
            seen.add(c)
            chosen.append(c)
    return np.array(chosen, dtype=np.int64)


def needle_query_tokens(w: Workload, t_lo: int = 0, t_hi: Optional[int] = None) -> np.ndarray:
    """Prefill tokens in [t_lo, t_hi) that carry the needle direction in every query head."""
    if not w.needle_query_every:
        return np.zeros(0, dtype=np.int64)
    t_hi = w.L if t_hi is None else t_hi
    r = draws(w.seed("needle") + 99, t_lo, t_hi - t_lo)
    return (np.nonzero((r % np.uint64(w.needle_query_every)) == 0)[0] + t_lo).astype(np.int64)


def chunk_offsets(w: Workload, b_lo=0, b_hi=None) -> np.ndarray:
    """[B, Nc, Hkv, d] fp32 per-chunk key offsets sigma * N(0,1) (exact in fp32 for sigma = 2^-k)."""
    b_hi = w.B if b_hi is None else b_hi
    raw = box(w.seed("offset"), (w.B, w.Nc, w.Hkv, w.d), (b_lo, 0, 0, 0), (b_hi, w.Nc, w.Hkv, w.d), "f32")
    return (raw * np.float32(w.chunk_offset_sigma)).astype(np.float32)


def host_tensor(w: Workload, tensor: str, lo: Sequence[int], hi: Sequence[int]) -> np.ndarray:
    """bf16 bit patterns of the box lo <= i < hi of q, K, V or dO, structure included.

    For prefill workloads the axes are (b, t, head, e); for decode q they are
    (0, query, head, e) and the memory K, V use (0, t, g, e).
    """
    dims = w.dims(tensor)
    x = box(w.seed(tensor), dims, lo, hi, "bf16")
    if x.size == 0:
        return x
    if tensor == "K" and not w.decode and w.chunk_offset_sigma:
        off = chunk_offsets(w, lo[0], hi[0])  # [b, Nc, Hkv, d]
        t = np.arange(lo[1], hi[1])
        chunk = t // w.S
        ok = chunk < w.Nc
        add = np.zeros(x.shape, dtype=np.float32)
        add[:, ok] = off[:, chunk[ok]][:, :, lo[2]:hi[2], lo[3]:hi[3]]
        x = np.where(ok[None, :, None, None], add_to_bf16(x, add), x)
    if w.needle_chunks and tensor == "K":
        ids = needle_chunk_ids(w)
        t = np.arange(lo[1], hi[1])
        for n, c in enumerate(ids):
            u = needle_direction(w, n if w.decode else 0)[lo[3]:hi[3]]
            sel = (t // w.S) == c
            if sel.any():
                x[:, sel] = add_to_bf16(x[:, sel], np.broadcast_to(u, x[:, sel].shape))
    if w.needle_chunks and tensor == "q":
        if w.decode:
            for qi in range(lo[1], hi[1]):
                u = needle_direction(w, qi)[lo[3]:hi[3]]
                x[:, qi - lo[1]] = add_to_bf16(x[:, qi - lo[1]], np.broadcast_to(u, x[:, qi - lo[1]].shape))
        else:
            toks = needle_query_tokens(w, lo[1], hi[1])
            if toks.size:
                u = needle_direction(w, 0)[lo[3]:hi[3]]
                sl = toks - lo[1]
                x[:, sl] = add_to_bf16(x[:, sl], np.broadcast_to(u, x[:, sl].shape))
    return x


def device_tensor(w: Workload, tensor: str, device="cuda"):
    """The whole tensor generated on the device (torch bf16), structure included."""
    import torch

    dims = w.dims(tensor)
    shape = dims[1:] if w.decode else dims
    out = torch.empty(shape, dtype=torch.bfloat16, device=device)
    lib = dev_lib()
    stream = ctypes.c_void_p(torch.cuda.current_stream(out.device).cuda_stream)
    rc = lib.synth_dev_fill_bf16(ctypes.c_void_p(out.data_ptr()), out.numel(), ctypes.c_uint64(w.seed(tensor)), 0,
                                 stream)
    if rc:
        raise RuntimeError(f"synth_dev_fill_bf16 failed ({rc})")
    d = w.d
    if tensor == "K" and not w.decode and w.chunk_offset_sigma:
        off = torch.from_numpy(chunk_offsets(w)).to(out.device)
        rc = lib.synth_dev_add_chunk_offsets(ctypes.c_void_p(out.data_ptr()), w.B, w.L, w.Hkv, w.d, w.S,
                                             ctypes.c_void_p(off.data_ptr()), stream)
        if rc:
            raise RuntimeError(f"synth_dev_add_chunk_offsets failed ({rc})")
        torch.cuda.current_stream(out.device).synchronize()
    rows_list, vecs_list = [], []
    if w.needle_chunks and tensor == "K":
        ids = needle_chunk_ids(w)
        H = w.Hkv
        for n, c in enumerate(ids):
            u = needle_direction(w, n if w.decode else 0)
            for b in range(1 if w.decode else w.B):
                t = np.arange(c * w.S, (c + 1) * w.S)
                rows = ((b * w.L + t)[:, None] * H + np.arange(H)[None, :]).reshape(-1)
                rows_list.append(rows)
                vecs_list.append(np.broadcast_to(u, (rows.size, d)))
    if w.needle_chunks and tensor == "q":
        if w.decode:
            for qi in range(w.Bq):
                u = needle_direction(w, qi)
                rows = qi * w.Hq + np.arange(w.Hq)
                rows_list.append(rows)
                vecs_list.append(np.broadcast_to(u, (rows.size, d)))
        else:
            toks = needle_query_tokens(w)
            u = needle_direction(w, 0)
            for b in range(w.B):
                rows = ((b * w.L + toks)[:, None] * w.Hq + np.arange(w.Hq)[None, :]).reshape(-1)
                rows_list.append(rows)
                vecs_list.append(u)
    if rows_list:
        for rows, vecs in zip(rows_list, vecs_list):
            rows_t = torch.from_numpy(np.ascontiguousarray(rows, dtype=np.int64)).to(out.device)
            v = np.asarray(vecs, dtype=np.float32)
            stride = 0 if v.ndim == 1 else d
            vecs_t = torch.from_numpy(np.ascontiguousarray(v)).to(out.device)
            rc = lib.synth_dev_add_rows(ctypes.c_void_p(out.data_ptr()), d, ctypes.c_void_p(rows_t.data_ptr()),
                                        ctypes.c_void_p(vecs_t.data_ptr()), rows_t.numel(), stride, stream)
            if rc:
                raise RuntimeError(f"synth_dev_add_rows failed ({rc})")
            torch.cuda.current_stream(out.device).synchronize()
    return out
