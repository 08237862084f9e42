"""Decode with the memory K, V kept in host memory (§3.2 "Inference": each step
reads only the summaries and the k selected chunks, so the token memory itself
can sit in the Grace memory behind the CPU-GPU link while the summaries stay in
HBM). The same kernels read the page-locked host pages at the host address:
results must be identical to a device-resident memory and match the oracle;
pageable memory must be refused on the host before any launch."""
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

INVALID = 1  # HSA_ERR_INVALID_ARG
NOALLOC_SCRATCH_BYTES = 8 << 20  # HSA_DECODE_NOALLOC_SCRATCH_BYTES


@pytest.fixture(scope="module", autouse=True)
def built():
    hsa.build()
    hsa.load()


def workload(topk=16, Hkv=1, Hq=16, d=128, L=64 * 520, Bq=33):
    return synth.Workload("dec-host", 71, B=1, L=L, S=64, Hq=Hq, Hkv=Hkv, d=d, topk=topk, Bq=Bq,
                          backward=False, decode=True, needle_chunks=Bq)


def memory(w):
    bits = {n: synth.host_tensor(w, n, (0, 0, 0, 0), w.dims(n)) for n in ("q", "K", "V")}
    qd = to_device_bf16(bits["q"][0])
    Kd = to_device_bf16(bits["K"][0])
    Vd = to_device_bf16(bits["V"][0])
    pshape = hsa.Shape(B=1, L=w.L, Hq=w.Hq, Hkv=w.Hkv, d=w.d, topk=w.topk)
    kbar32, _ = hsa.chunk_pool(pshape, Kd.view(1, w.L, w.Hkv, w.d), want_bf16=False)
    return bits, qd, Kd, Vd, kbar32.view(w.Nc, w.Hkv, w.d)


def outputs_equal(a, b):
    for x, y in zip(a, b):
        assert torch.equal(x, y)


@pytest.mark.parametrize("kind", ["pinned", "registered"])
@pytest.mark.parametrize("topk", [16, 32])  # indexed scan (k <= 16) and the CUDA-core scan
def test_host_memory_decode_identical_to_device_memory(kind, topk):
    w = workload(topk=topk)
    bits, qd, Kd, Vd, kb = memory(w)
    if kind == "pinned":
        Kh = Kd.cpu().pin_memory()
        Vh = Vd.cpu().pin_memory()
        assert Kh.is_pinned() and Vh.is_pinned()
    else:  # ordinary host pages, page-locked and mapped afterwards
        Kh, Vh = Kd.cpu(), Vd.cpu()
        for t in (Kh, Vh):
            rc = torch.cuda.cudart().cudaHostRegister(t.data_ptr(), t.numel() * t.element_size(), 2)
            assert int(rc) == 0, rc
    try:
        dshape = hsa.DecodeShape(Bq=w.Bq, Hq=w.Hq, Hkv=w.Hkv, d=w.d, n_chunks=w.Nc, topk=w.topk)
        index = hsa.decode_index(dshape, kb)
        ref_dev = [t.clone() for t in hsa.decode_indexed(dshape, qd, Kd, Vd, kb, index)]
        got = [t.clone() for t in hsa.decode_indexed(dshape, qd, Kh, Vh, kb, index)]
        exact_dev = [t.clone() for t in hsa.decode(dshape, qd, Kd, Vd, kb)]
        exact = [t.clone() for t in hsa.decode(dshape, qd, Kh, Vh, kb)]
        torch.cuda.synchronize()
        outputs_equal(got, ref_dev)
        outputs_equal(exact, exact_dev)
        if hsa.decode_workspace_size(dshape) <= NOALLOC_SCRATCH_BYTES:
            O, idx, s_sel, wts = (torch.empty_like(t) for t in exact)
            hsa.decode_noalloc(dshape, qd, Kh, Vh, kb, O, idx, s_sel, wts)
            torch.cuda.synchronize()
            outputs_equal((O, idx, s_sel, wts), exact_dev)
    finally:
        if kind == "registered":
            for t in (Kh, Vh):
                torch.cuda.cudart().cudaHostUnregister(t.data_ptr())
    # and against the oracle, from the host-memory run
    K = synth.bf16_to_f64(bits["K"])[0]
    V = synth.bf16_to_f64(bits["V"])[0]
    kb64 = oracle.pool(K[None], w.S, f32=True)[0]
    ref = oracle.decode(synth.bf16_to_f64(bits["q"])[0], K, V, kb64, w.S, w.topk, f32=True)
    assert np.array_equal(got[1].cpu().numpy(), ref["idx"])
    assert np.array_equal(got[2].cpu().numpy(), ref["s_sel"].astype(np.float32))
    assert_close("decode w", got[3].cpu().numpy(), ref["w"], max_abs=1e-5, rel=1e-5)
    assert_close("decode O", bf16_tensor_to_f64(got[0]), ref["O"])


def test_pageable_host_memory_is_refused_before_launch():
    w = workload(topk=8, Hq=8, d=64, L=64 * 40, Bq=4)
    _, qd, Kd, Vd, kb = memory(w)
    Kp, Vp = Kd.cpu(), Vd.cpu()  # ordinary pageable pages
    assert not Kp.is_pinned()
    dshape = hsa.DecodeShape(Bq=w.Bq, Hq=w.Hq, Hkv=w.Hkv, d=w.d, n_chunks=w.Nc, topk=w.topk)
    index = hsa.decode_index(dshape, kb)
    for call in (lambda: hsa.decode_indexed(dshape, qd, Kp, Vd, kb, index),
                 lambda: hsa.decode_indexed(dshape, qd, Kd, Vp, kb, index),
                 lambda: hsa.decode(dshape, qd, Kp, Vp, kb)):
        with pytest.raises(hsa.HsaError) as e:
            call()
        assert e.value.status == INVALID
    outs = [torch.empty((w.Bq, w.Hkv, w.topk), dtype=t, device="cuda")
            for t in (torch.int32, torch.float32, torch.float32)]
    with pytest.raises(hsa.HsaError) as e:
        hsa.decode_noalloc(dshape, qd, Kp, Vp, kb, torch.empty_like(qd), *outs)
    assert e.value.status == INVALID
    torch.cuda.synchronize()
