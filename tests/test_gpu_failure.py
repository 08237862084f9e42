"""Failure detection on the device without a fault: a wait that nothing ever
completes gives up after its limit, records the timeout in a status word that
hsa_device_check reports once, and leaves the context usable (a selection
computed afterwards still matches the oracle)."""
import time

import numpy as np
import pytest

import oracle
import synth
from hsa_cases import bf16_tensor_to_f64

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover - collected on CPU only with -m gpu
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2504_16795_gb300 as hsa  # noqa: E402

OK, TIMEOUT, INVALID = 0, 5, 1


@pytest.fixture(scope="module", autouse=True)
def built():
    hsa.build()
    hsa.load()


def test_a_wait_nothing_completes_gives_up_and_is_reported_once():
    lib = hsa.load()
    assert lib.hsa_device_check() == OK  # clears anything earlier tests left
    t0 = time.time()
    hsa.selftest_wait_timeout(1_000_000)  # 1 ms
    assert lib.hsa_device_check() == TIMEOUT
    assert time.time() - t0 < 10.0
    assert lib.hsa_device_check() == OK  # reported once, then cleared


def test_the_limit_is_validated_before_any_launch():
    lib = hsa.load()
    before = lib.hsa_kernel_launches()
    assert lib.hsa_selftest_wait_timeout(0, None) == INVALID
    assert lib.hsa_selftest_wait_timeout(2_000_000_000, None) == INVALID
    assert lib.hsa_kernel_launches() == before


def test_the_context_stays_usable_after_a_wait_gave_up():
    hsa.selftest_wait_timeout(1_000_000)
    assert hsa.load().hsa_device_check() == TIMEOUT
    w = synth.WORKLOADS[1]
    shape = hsa.Shape(B=w.B, L=w.L, Hq=w.Hq, Hkv=w.Hkv, d=w.d, S=w.S, topk=w.topk)
    q = synth.device_tensor(w, "q")
    K = synth.device_tensor(w, "K")
    kbar32, _ = hsa.chunk_pool(shape, K)
    idx, s_sel = hsa.select_topk(shape, q, kbar32)
    hsa.device_check()
    kb = oracle.pool(bf16_tensor_to_f64(K), w.S, f32=True)
    assert np.array_equal(kbar32.cpu().numpy(), kb.astype(np.float32))
    o_idx, _, _ = oracle.select(bf16_tensor_to_f64(q), kb, w.S, w.topk, f32=True)
    assert np.array_equal(idx.cpu().numpy(), o_idx)
