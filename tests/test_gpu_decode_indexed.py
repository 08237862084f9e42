"""hsa_decode_indexed (tensor-core scan of a prebuilt memory index, exact
rescoring) against the CPU oracle on small memories and against hsa_decode
(CUDA-core exact scan) at the 2^26-token memory: identical indices and scores,
weights and outputs within tolerance."""
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


@pytest.fixture(scope="module", autouse=True)
def built():
    hsa.build()
    hsa.load()


def small_memory(w, bits=None):
    T, Nc, d = w.L, w.Nc, w.d
    bits = bits or {n: synth.host_tensor(w, n, (0, 0, 0, 0), w.dims(n)) for n in ("q", "K", "V")}
    qd = to_device_bf16(bits["q"][0])
    Kmem = to_device_bf16(bits["K"][0])
    Vmem = to_device_bf16(bits["V"][0])
    pshape = hsa.Shape(B=1, L=T, Hq=w.Hq, Hkv=w.Hkv, d=d, topk=w.topk)
    kbar32, _ = hsa.chunk_pool(pshape, Kmem.view(1, T, w.Hkv, d), want_bf16=False)
    return bits, qd, Kmem, Vmem, kbar32.view(Nc, w.Hkv, d)


def check_against_oracle(w, bits=None, inner="softmax", weights="softmax", exact=False):
    bits, qd, Kmem, Vmem, kbar32 = small_memory(w, bits)
    dshape = hsa.DecodeShape(Bq=w.Bq, Hq=w.Hq, Hkv=w.Hkv, d=w.d, n_chunks=w.Nc, topk=w.topk, inner=inner,
                             weights=weights)
    if exact:
        O, idx, s_sel, wts = hsa.decode(dshape, qd, Kmem, Vmem, kbar32)
    else:
        index = hsa.decode_index(dshape, kbar32)
        O, idx, s_sel, wts = hsa.decode_indexed(dshape, qd, Kmem, Vmem, kbar32, index)
    torch.cuda.synchronize()
    K = synth.bf16_to_f64(bits["K"])[0]
    V = synth.bf16_to_f64(bits["V"])[0]
    kb = oracle.pool(K[None], w.S, f32=True)[0]
    ref = oracle.decode(synth.bf16_to_f64(bits["q"])[0], K, V, kb, w.S, w.topk, f32=True, inner=inner,
                        weights=weights)
    assert np.array_equal(idx.cpu().numpy(), ref["idx"])
    assert np.array_equal(s_sel.cpu().numpy(), ref["s_sel"].astype(np.float32))
    assert_close("decode w", wts.cpu().numpy(), ref["w"], max_abs=1e-5, rel=1e-5)
    assert_close("decode O", bf16_tensor_to_f64(O), ref["O"])
    return idx


CASES = {
    "d64 k8 two groups": dict(L=64 * 300, Hq=8, Hkv=2, d=64, topk=8, Bq=70),
    "d128 k16 one group": dict(L=64 * 520, Hq=16, Hkv=1, d=128, topk=16, Bq=33),
    "d128 k4 G2": dict(L=64 * 130 + 17, Hq=4, Hkv=2, d=128, topk=4, Bq=129),
    # at most 64 queries and groups of 8 columns: two scan threads per row
    "d128 k4 two threads per row": dict(L=64 * 700, Hq=8, Hkv=1, d=128, topk=4, Bq=64),
    "d64 k2 G2 two threads per row, ragged": dict(L=64 * 250 + 9, Hq=4, Hkv=2, d=64, topk=2, Bq=17),
}


@pytest.mark.parametrize("name", list(CASES))
def test_indexed_decode_matches_oracle(name):
    kw = CASES[name]
    w = synth.Workload("dec-ix", 61, B=1, S=64, backward=False, decode=True, needle_chunks=kw["Bq"], **kw)
    check_against_oracle(w)


@pytest.mark.parametrize("exact", [False, True])
@pytest.mark.parametrize("variant", [("softmax1", "softmax"), ("softmax", "stick"), ("softmax1", "stick")])
def test_decode_variants_match_oracle(variant, exact):
    # softmax-off-by-one inside chunks (§3.1.2) and stick-breaking chunk weights (§3.1.1)
    kw = CASES["d64 k8 two groups"]
    w = synth.Workload("dec-var", 63, B=1, S=64, backward=False, decode=True, needle_chunks=kw["Bq"], **kw)
    check_against_oracle(w, inner=variant[0], weights=variant[1], exact=exact)


@pytest.mark.parametrize("topk", [8, 4])
def test_indexed_decode_equal_summaries_take_the_exact_path(topk):
    # every chunk of the memory equal: every score of a query ties, the
    # per-range candidate buffers overflow and the merge scores whole ranges
    # (k = 4: two scan threads per row)
    w = synth.Workload("dec-eq", 62, B=1, L=64 * 200, S=64, Hq=8, Hkv=1, d=64, topk=topk, backward=False,
                       decode=True, Bq=9)
    bits = {n: synth.host_tensor(w, n, (0, 0, 0, 0), w.dims(n)) for n in ("q", "K", "V")}
    K = bits["K"]
    for c in range(1, w.Nc):
        K[:, c * 64:(c + 1) * 64] = K[:, 0:64]
    idx = check_against_oracle(w, bits)
    assert (idx[:, 0, :].cpu().numpy() == np.arange(topk - 1, -1, -1)).all()


def test_indexed_decode_64m_memory_matches_exact_decode():
    w = synth.WORKLOADS[5]
    T, Nc, d = w.L, w.Nc, w.d
    dshape = hsa.DecodeShape(Bq=w.Bq, Hq=w.Hq, Hkv=w.Hkv, d=d, n_chunks=Nc, topk=w.topk)
    pshape = hsa.Shape(B=1, L=T, Hq=w.Hq, Hkv=w.Hkv, d=d, topk=w.topk)
    Kmem = synth.device_tensor(w, "K")
    Vmem = synth.device_tensor(w, "V")
    qd = synth.device_tensor(w, "q")
    kbar32, _ = hsa.chunk_pool(pshape, Kmem.view(1, T, w.Hkv, d), want_bf16=False)
    kbar32 = kbar32.view(Nc, w.Hkv, d)
    O0, idx0, s0, w0 = hsa.decode(dshape, qd, Kmem, Vmem, kbar32)
    index = hsa.decode_index(dshape, kbar32)
    O1, idx1, s1, w1 = hsa.decode_indexed(dshape, qd, Kmem, Vmem, kbar32, index)
    torch.cuda.synchronize()
    assert np.array_equal(idx1.cpu().numpy(), idx0.cpu().numpy())
    assert np.array_equal(s1.cpu().numpy(), s0.cpu().numpy())
    assert_close("w", w1.cpu().numpy(), w0.cpu().numpy(), max_abs=1e-6, rel=1e-6)
    assert_close("O", bf16_tensor_to_f64(O1), bf16_tensor_to_f64(O0), max_abs=1e-2, rel=1e-3)
    needles = synth.needle_chunk_ids(w)
    got = idx1.cpu().numpy()
    for b in range(w.Bq):
        assert needles[b] in got[b, 0], b
