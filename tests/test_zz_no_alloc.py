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
    for call, q in enumerate(queries):
        O = torch.full_like(q, float("nan"))
        idx = torch.full(res, 12345, dtype=torch.int32, device=dev)
        s_sel = torch.full(res, float("nan"), dtype=torch.float32, device=dev)
        wts = torch.full(res, float("nan"), dtype=torch.float32, device=dev)
        hsa.decode_noalloc(dshape, q, K, V, kbar32, O, idx, s_sel, wts)
        rO, ridx, rs, rw = hsa.decode(dshape, q, K, V, kbar32)
        torch.cuda.synchronize()
        hsa.device_check()
        assert np.array_equal(idx.cpu().numpy(), ridx.cpu().numpy()), call
        assert np.array_equal(s_sel.cpu().numpy(), rs.cpu().numpy()), call
        assert_close(f"call {call} w", wts.cpu().numpy(), rw.cpu().numpy(), max_abs=1e-5, rel=1e-5)
        assert_close(f"call {call} O", bf16_tensor_to_f64(O), bf16_tensor_to_f64(rO))
