"""Failure detection on the device without a fault: a wait that nothing ever
completes gives up after its limit and records the timeout in the status word
at the head of the workspace of its call; hsa_check of that workspace reports
it once, a workspace used on another stream stays clean, and the context
stays usable (a selection computed afterwards still matches the oracle)."""
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

OK, INVALID, WORKSPACE, TIMEOUT = 0, 1, 3, 5


@pytest.fixture(scope="module", autouse=True)
def built():
    hsa.build()
    hsa.load()


def raw_check(ws):
    return hsa.load().hsa_check(hsa.binding._ptr(ws), ws.numel(), hsa.binding._stream(ws.device))


def test_a_wait_nothing_completes_gives_up_and_is_reported_once():
    ws = hsa.new_workspace(hsa.status_bytes(), "cuda")
    assert raw_check(ws) == OK
    t0 = time.time()
    hsa.selftest_wait_timeout(1_000_000, ws)  # 1 ms
    assert raw_check(ws) == TIMEOUT
    assert time.time() - t0 < 10.0
    assert raw_check(ws) == OK  # reported once, then cleared


def test_each_workspace_reports_only_its_own_calls():
    # two streams, each with its own workspace: the self-test times out on
    # stream a while a real selection runs on stream b
    w = synth.WORKLOADS[1]
    shape = hsa.Shape(B=w.B, L=w.L, Hq=w.Hq, Hkv=w.Hkv, d=w.d, S=w.S, topk=w.topk)
    q = synth.device_tensor(w, "q")
    K = synth.device_tensor(w, "K")
    kbar32, _ = hsa.chunk_pool(shape, K)
    ws_a = hsa.new_workspace(hsa.status_bytes(), "cuda")
    ws_b = hsa.new_workspace(hsa.workspace_size(hsa.HSA_OP_SELECT, shape), "cuda")
    torch.cuda.synchronize()
    sa, sb = torch.cuda.Stream(), torch.cuda.Stream()
    with torch.cuda.stream(sa):
        hsa.selftest_wait_timeout(2_000_000, ws_a)
    with torch.cuda.stream(sb):
        idx, _ = hsa.select_topk(shape, q, kbar32, ws=ws_b)
    with torch.cuda.stream(sb):
        assert raw_check(ws_b) == OK
    with torch.cuda.stream(sa):
        assert raw_check(ws_a) == TIMEOUT
        assert raw_check(ws_a) == OK
    torch.cuda.synchronize()
    o_idx, _, _ = oracle.select(bf16_tensor_to_f64(q), oracle.pool(bf16_tensor_to_f64(K), w.S, f32=True), w.S,
                                w.topk, f32=True)
    assert np.array_equal(idx.cpu().numpy(), o_idx)


def test_the_limit_and_workspace_are_validated_before_any_launch():
    lib = hsa.load()
    ws = hsa.new_workspace(hsa.status_bytes(), "cuda")
    p, n, st = hsa.binding._ptr(ws), ws.numel(), hsa.binding._stream(ws.device)
    before = lib.hsa_kernel_launches()
    assert lib.hsa_selftest_wait_timeout(0, p, n, st) == INVALID
    assert lib.hsa_selftest_wait_timeout(2_000_000_000, p, n, st) == INVALID
    assert lib.hsa_selftest_wait_timeout(1000, None, n, st) == WORKSPACE
    assert lib.hsa_selftest_wait_timeout(1000, p, n - 1, st) == WORKSPACE
    assert lib.hsa_check(None, n, st) == INVALID
    assert lib.hsa_check(p, n - 1, st) == INVALID
    assert lib.hsa_kernel_launches() == before


def test_the_context_stays_usable_after_a_wait_gave_up():
    ws0 = hsa.new_workspace(hsa.status_bytes(), "cuda")
    hsa.selftest_wait_timeout(1_000_000, ws0)
    assert raw_check(ws0) == TIMEOUT
    w = synth.WORKLOADS[1]
    shape = hsa.Shape(B=w.B, L=w.L, Hq=w.Hq, Hkv=w.Hkv, d=w.d, S=w.S, topk=w.topk)
    q = synth.device_tensor(w, "q")
    K = synth.device_tensor(w, "K")
    kbar32, _ = hsa.chunk_pool(shape, K)
    ws = hsa.new_workspace(hsa.workspace_size(hsa.HSA_OP_SELECT, shape), "cuda")
    idx, s_sel = hsa.select_topk(shape, q, kbar32, ws=ws)
    hsa.check(ws)
    kb = oracle.pool(bf16_tensor_to_f64(K), w.S, f32=True)
    assert np.array_equal(kbar32.cpu().numpy(), kb.astype(np.float32))
    o_idx, _, _ = oracle.select(bf16_tensor_to_f64(q), kb, w.S, w.topk, f32=True)
    assert np.array_equal(idx.cpu().numpy(), o_idx)
