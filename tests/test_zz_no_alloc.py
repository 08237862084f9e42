"""hsa_decode_noalloc (library-owned scratch, no workspace argument) against
hsa_decode on the same seeded inputs, through the C ABI, on two calls in a row.

Kept in a file of its own that sorts last, so that it runs both alone in a
fresh process and after every other GPU test has used the device."""
import numpy as np
import pytest

import synth
from hsa_cases import assert_close, bf16_tensor_to_f64, to_device_bf16

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover - collected on CPU only with -m gpu
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2504_16795_gb300 as hsa  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def built():
    hsa.build()
    hsa.load()


def test_decode_noalloc_matches_decode_on_consecutive_calls():
    # a memory of 300 chunks (ragged last scan tile), 70 queries (two query
    # tiles, the second ragged), two groups of four heads
    w = synth.Workload("dec-noalloc", 53, B=1, L=64 * 300, S=64, Hq=8, Hkv=2, d=64, topk=8, backward=False,
                       decode=True, Bq=70, needle_chunks=70)
    T, Nc, d = w.L, w.Nc, w.d
    K = to_device_bf16(synth.host_tensor(w, "K", (0, 0, 0, 0), w.dims("K"))[0])
    V = to_device_bf16(synth.host_tensor(w, "V", (0, 0, 0, 0), w.dims("V"))[0])
    pshape = hsa.Shape(B=1, L=T, Hq=w.Hq, Hkv=w.Hkv, d=d, topk=w.topk)
    kbar32, _ = hsa.chunk_pool(pshape, K.view(1, T, w.Hkv, d), want_bf16=False)
    kbar32 = kbar32.view(Nc, w.Hkv, d)
    dshape = hsa.DecodeShape(Bq=w.Bq, Hq=w.Hq, Hkv=w.Hkv, d=d, n_chunks=Nc, topk=w.topk)
    assert hsa.decode_workspace_size(dshape) <= 8 << 20

    qbits = synth.host_tensor(w, "q", (0, 0, 0, 0), w.dims("q"))[0]
    queries = [to_device_bf16(qbits), to_device_bf16(qbits[::-1].copy())]  # two different query batches
    dev = queries[0].device
    res = (w.Bq, w.Hkv, w.topk)
    refs = [hsa.decode(dshape, q, K, V, kbar32) for q in queries]
    outs = []
    for q in queries:
        outs.append((torch.full_like(q, float("nan")), torch.full(res, 12345, dtype=torch.int32, device=dev),
                     torch.full(res, float("nan"), dtype=torch.float32, device=dev),
                     torch.full(res, float("nan"), dtype=torch.float32, device=dev)))
    # a first call loads the kernels (lazy module loading may take device memory once)
    warm = [torch.empty_like(t) for t in outs[0]]
    hsa.decode_noalloc(dshape, queries[0], K, V, kbar32, *warm)
    torch.cuda.synchronize()
    free0, alloc0 = torch.cuda.mem_get_info(dev)[0], torch.cuda.memory_allocated(dev)
    for q, o in zip(queries, outs):
        hsa.decode_noalloc(dshape, q, K, V, kbar32, *o)
    torch.cuda.synchronize()
    # the calls took no device memory: neither through torch nor from the driver
    assert torch.cuda.memory_allocated(dev) == alloc0
    assert torch.cuda.mem_get_info(dev)[0] == free0
    for call, (o, r) in enumerate(zip(outs, refs)):
        # the same kernels on the same inputs: identical results
        for name, a, b in zip(("O", "idx", "s_sel", "w"), o, r):
            assert torch.equal(a, b), f"call {call}: {name} differs from hsa_decode"
    # and hsa_decode itself against the expected properties of the query batch
    assert_close("w sums to 1", outs[1][3].sum(-1).cpu().numpy().astype(np.float64), np.ones((w.Bq, w.Hkv)),
                 max_abs=1e-5, rel=1e-5)
    assert np.isfinite(bf16_tensor_to_f64(outs[1][0])).all()


def test_decode_noalloc_over_an_empty_memory_takes_null_memory_pointers():
    # no chunk in the memory: nothing is selected and the output is 0, as hsa_decode gives
    dshape = hsa.DecodeShape(Bq=3, Hq=8, Hkv=2, d=64, n_chunks=0, topk=4)
    q = torch.randn((3, 8, 64), device="cuda").to(torch.bfloat16)
    outs = (torch.full_like(q, float("nan")), torch.full((3, 2, 4), 7, dtype=torch.int32, device="cuda"),
            torch.zeros((3, 2, 4), dtype=torch.float32, device="cuda"),
            torch.full((3, 2, 4), float("nan"), dtype=torch.float32, device="cuda"))
    hsa.decode_noalloc(dshape, q, None, None, None, *outs)
    ref = hsa.decode(dshape, q, None, None, None)
    torch.cuda.synchronize()
    for name, a, b in zip(("O", "idx", "s_sel", "w"), outs, ref):
        assert torch.equal(a, b), name
    assert (outs[1] == -1).all() and (outs[0].float() == 0).all() and (outs[3] == 0).all()
