"""A decode memory grown by appends (§3.2 "Inference": tokens join the memory as
they are decoded, a chunk is summarised once complete, only completed chunks are
selectable). After every append the memory, its summaries and its decode index
must be bit-identical to building them at once from the same tokens, and decode
over it must match the oracle on the memory's completed chunks."""
import numpy as np
import pytest

import oracle
import synth
from hsa_cases import assert_close, bf16_tensor_to_f64, to_device_bf16

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover - collected on CPU only with -m gpu
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2504_16795_gb300 as hsa  # noqa: E402

S = 64


@pytest.fixture(scope="module", autouse=True)
def built():
    hsa.build()
    hsa.load()


def tokens(Hq, Hkv, d, topk, T, Bq, seed=81):
    w = synth.Workload("dec-grow", seed, B=1, L=T, S=S, Hq=Hq, Hkv=Hkv, d=d, topk=topk, Bq=Bq, backward=False,
                       decode=True, needle_chunks=Bq)
    return w, {n: synth.host_tensor(w, n, (0, 0, 0, 0), w.dims(n))[0] for n in ("q", "K", "V")}


class Memory:
    """A memory of `cap` chunks on the device (or K, V in pinned host memory), its
    summaries and, for topk <= 16, its decode index."""

    def __init__(self, Hq, Hkv, d, topk, cap, host=False):
        self.Hq, self.Hkv, self.d, self.topk, self.cap = Hq, Hkv, d, topk, cap
        shape = (cap * S, Hkv, d)
        if host:
            self.K = torch.zeros(shape, dtype=torch.bfloat16).pin_memory()
            self.V = torch.zeros(shape, dtype=torch.bfloat16).pin_memory()
        else:
            self.K = torch.zeros(shape, dtype=torch.bfloat16, device="cuda")
            self.V = torch.zeros(shape, dtype=torch.bfloat16, device="cuda")
        self.kbar32 = torch.zeros((cap, Hkv, d), dtype=torch.float32, device="cuda")
        self.T = 0
        self.index = hsa.decode_index(self.shape(Bq=1), self.kbar32)

    def shape(self, Bq, n_chunks=None):
        return hsa.DecodeShape(Bq=Bq, Hq=self.Hq, Hkv=self.Hkv, d=self.d, topk=self.topk,
                               n_chunks=self.T // S if n_chunks is None else n_chunks, capacity_chunks=self.cap)

    def append(self, Kn, Vn):
        self.T = hsa.memory_append(self.shape(Bq=1), self.T, Kn, Vn, self.K, self.V, self.kbar32, self.index)


def check_state(mem, bits):
    """The grown memory against everything built at once from its tokens."""
    T, Nc = mem.T, mem.T // S
    torch.cuda.synchronize()
    K = to_device_bf16(bits["K"][:T])
    V = to_device_bf16(bits["V"][:T])
    assert torch.equal(mem.K[:T].cuda(), K) and torch.equal(mem.V[:T].cuda(), V)
    if Nc == 0:
        return
    pshape = hsa.Shape(B=1, L=Nc * S, Hq=mem.Hq, Hkv=mem.Hkv, d=mem.d, topk=mem.topk)
    kb_once, _ = hsa.chunk_pool(pshape, K[:Nc * S].reshape(1, Nc * S, mem.Hkv, mem.d).contiguous(),
                                want_bf16=False)
    assert torch.equal(mem.kbar32[:Nc], kb_once.view(Nc, mem.Hkv, mem.d))
    assert not mem.kbar32[Nc:].any()  # chunks not yet complete stay untouched
    if mem.index is not None:
        once = hsa.decode_index(mem.shape(Bq=1), kb_once.view(Nc, mem.Hkv, mem.d).contiguous())
        assert torch.equal(mem.index, once)


def check_decode(mem, bits, w):
    T, Nc = mem.T, mem.T // S
    q = to_device_bf16(bits["q"])
    dshape = mem.shape(Bq=w.Bq)
    if mem.index is not None:
        O, idx, s_sel, wts = hsa.decode_indexed(dshape, q, mem.K, mem.V, mem.kbar32, mem.index)
    else:
        O, idx, s_sel, wts = hsa.decode(dshape, q, mem.K, mem.V, mem.kbar32)
    torch.cuda.synchronize()
    # a memory that does not grow, built at once from the completed chunks
    fixed = hsa.DecodeShape(Bq=w.Bq, Hq=mem.Hq, Hkv=mem.Hkv, d=mem.d, topk=mem.topk, n_chunks=Nc)
    Kd = to_device_bf16(bits["K"][:Nc * S])
    Vd = to_device_bf16(bits["V"][:Nc * S])
    if Nc > 0:
        pshape = hsa.Shape(B=1, L=Nc * S, Hq=mem.Hq, Hkv=mem.Hkv, d=mem.d, topk=mem.topk)
        kb, _ = hsa.chunk_pool(pshape, Kd.view(1, Nc * S, mem.Hkv, mem.d), want_bf16=False)
        kb = kb.view(Nc, mem.Hkv, mem.d)
        ix = hsa.decode_index(fixed, kb)
        ref_gpu = hsa.decode_indexed(fixed, q, Kd, Vd, kb, ix)
        for a, b in zip((O, idx, s_sel, wts), ref_gpu):
            assert torch.equal(a, b)
    K64 = synth.bf16_to_f64(bits["K"][:Nc * S])
    V64 = synth.bf16_to_f64(bits["V"][:Nc * S])
    kb64 = oracle.pool(K64[None], S, f32=True)[0]
    ref = oracle.decode(synth.bf16_to_f64(bits["q"]), K64, V64, kb64, S, mem.topk, f32=True)
    assert np.array_equal(idx.cpu().numpy(), ref["idx"])
    assert np.array_equal(s_sel.cpu().numpy(), ref["s_sel"].astype(np.float32))
    assert_close("w", wts.cpu().numpy(), ref["w"], max_abs=1e-5, rel=1e-5)
    assert_close("O", bf16_tensor_to_f64(O), ref["O"])


# ragged appends: single tokens across a chunk boundary, pieces that complete
# several chunks at once, pieces ending mid-chunk
PIECES = [1, 62, 1, 1, 64, 200, 7] + [1] * 70 + [3000, 640, 129, 5000]


@pytest.mark.parametrize("cfg", [dict(Hq=8, Hkv=2, d=64, topk=8), dict(Hq=16, Hkv=1, d=128, topk=16),
                                 dict(Hq=4, Hkv=2, d=128, topk=24)])
def test_grown_memory_equals_memory_built_at_once(cfg):
    cap = 200
    T_all = sum(PIECES)
    assert T_all <= cap * S
    w, bits = tokens(T=T_all, Bq=21, **cfg)
    mem = Memory(cap=cap, **cfg)
    assert (mem.index is None) == (cfg["topk"] > 16)
    t = 0
    for i, n in enumerate(PIECES):
        mem.append(to_device_bf16(bits["K"][t:t + n]), to_device_bf16(bits["V"][t:t + n]))
        t += n
        assert mem.T == t
        if i in (0, 2, 6, len(PIECES) - 3) or i == len(PIECES) - 1:
            check_state(mem, bits)
            check_decode(mem, bits, w)


def test_prefill_written_in_place_then_appended():
    # a prefill stores its keys and values straight into the memory, then the
    # append pools them with K_new aliasing the memory's own rows
    cfg = dict(Hq=8, Hkv=1, d=128, topk=8)
    w, bits = tokens(T=64 * 90 + 17, Bq=9, seed=83, **cfg)
    mem = Memory(cap=128, **cfg)
    first = 64 * 30 + 5
    mem.append(to_device_bf16(bits["K"][:first]), to_device_bf16(bits["V"][:first]))
    rest = w.L - first
    mem.K[first:first + rest] = to_device_bf16(bits["K"][first:])
    mem.V[first:first + rest] = to_device_bf16(bits["V"][first:])
    mem.append(mem.K[first:first + rest], mem.V[first:first + rest])
    check_state(mem, bits)
    check_decode(mem, bits, w)


def test_memory_grown_in_host_memory():
    cfg = dict(Hq=8, Hkv=2, d=64, topk=8)
    w, bits = tokens(T=64 * 150 + 33, Bq=12, seed=85, **cfg)
    mem = Memory(cap=160, host=True, **cfg)
    t = 0
    for n in (70, 1, 1, 4000, 129, w.L - 4201):
        mem.append(to_device_bf16(bits["K"][t:t + n]), to_device_bf16(bits["V"][t:t + n]))
        t += n
    check_state(mem, bits)
    check_decode(mem, bits, w)


def test_prefill_size_append_equals_building_at_once():
    # a 2^20-token prefill (the long prefill workload's memory) appended in three
    # ragged pieces, against pooling and indexing it at once
    w = synth.WORKLOADS[5].with_(L=1 << 20)
    T, Hkv, d = w.L, w.Hkv, w.d
    Kn = synth.device_tensor(w, "K")
    Vn = synth.device_tensor(w, "V")
    mem = Memory(Hq=w.Hq, Hkv=Hkv, d=d, topk=w.topk, cap=T // S + 3)
    for lo, hi in ((0, 12345), (12345, 12345 + 64 * 1000 + 1), (12345 + 64 * 1000 + 1, T)):
        mem.append(Kn[lo:hi], Vn[lo:hi])
    torch.cuda.synchronize()
    assert mem.T == T
    assert torch.equal(mem.K[:T], Kn) and torch.equal(mem.V[:T], Vn)
    pshape = hsa.Shape(B=1, L=T, Hq=w.Hq, Hkv=Hkv, d=d, topk=w.topk)
    kb_once, _ = hsa.chunk_pool(pshape, Kn.view(1, T, Hkv, d), want_bf16=False)
    assert torch.equal(mem.kbar32[:T // S], kb_once.view(T // S, Hkv, d))
    once = hsa.decode_index(mem.shape(Bq=1), kb_once.view(T // S, Hkv, d).contiguous())
    assert torch.equal(mem.index, once)
