"""The hot path captured in a CUDA graph and replayed (how a training or serving
loop removes its per-call launch cost): every entry point must be capturable,
and replays must reproduce the eager results bit for bit (the kernels are
deterministic), including the decode chain, whose kernels start as programmatic
dependents of the kernel before them."""
import pytest

import synth
from hsa_cases import to_device_bf16

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover - collected on CPU only with -m gpu
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2504_16795_gb300 as hsa  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def built():
    hsa.build()
    hsa.load()


def capture(fn):
    """Warm up on a side stream, then capture fn() into a graph; returns (graph, outputs)."""
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        fn()
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, capture_error_mode="relaxed"):
        out = fn()
    return g, out


@pytest.mark.parametrize("weights", ["softmax", "stick"])
def test_prefill_step_replays_bit_exactly(weights):
    w = synth.WORKLOADS[2].with_(B=2, L=2048 + 37)
    shape = hsa.Shape(B=w.B, L=w.L, Hq=w.Hq, Hkv=w.Hkv, d=w.d, S=w.S, topk=w.topk, weights=weights)
    X = {n: to_device_bf16(synth.host_tensor(w, n, (0, 0, 0, 0), w.dims(n))) for n in ("q", "K", "V", "dO")}
    wss = hsa.Workspaces(shape, X["q"].device)

    def step():
        fwd = hsa.hsa_forward_path(shape, X["q"], X["K"], X["V"], wss)
        dq, dK, dV = hsa.hsa_backward_path(shape, X["q"], X["K"], X["V"], fwd, X["dO"], wss)
        return fwd["idx"], fwd["O"], dq, dK, dV

    eager = [t.clone() for t in step()]
    g, out = capture(step)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    wss.check()
    for a, b in zip(out, eager):
        assert torch.equal(a, b)


def test_decode_chain_replays_bit_exactly():
    w = synth.Workload("dec-graph", 91, B=1, L=64 * 700, S=64, Hq=8, Hkv=1, d=128, topk=8, Bq=64,
                       backward=False, decode=True, needle_chunks=64)
    bits = {n: synth.host_tensor(w, n, (0, 0, 0, 0), w.dims(n)) for n in ("q", "K", "V")}
    q, K, V = (to_device_bf16(bits[n][0]) for n in ("q", "K", "V"))
    kb, _ = hsa.chunk_pool(hsa.Shape(B=1, L=w.L, Hq=w.Hq, Hkv=w.Hkv, d=w.d, topk=w.topk),
                           K.view(1, w.L, w.Hkv, w.d), want_bf16=False)
    kb = kb.view(w.Nc, w.Hkv, w.d)
    ds = hsa.DecodeShape(Bq=w.Bq, Hq=w.Hq, Hkv=w.Hkv, d=w.d, n_chunks=w.Nc, topk=w.topk)
    index = hsa.decode_index(ds, kb)
    outs = [torch.empty_like(q), torch.empty((w.Bq, w.Hkv, w.topk), dtype=torch.int32, device=q.device),
            torch.empty((w.Bq, w.Hkv, w.topk), dtype=torch.float32, device=q.device),
            torch.empty((w.Bq, w.Hkv, w.topk), dtype=torch.float32, device=q.device)]
    nws = hsa.load().hsa_decode_indexed_workspace_size(__import__("ctypes").byref(ds.c()))
    ws = hsa.new_workspace(int(nws), q.device)

    def call():
        return hsa.decode_indexed(ds, q, K, V, kb, index, *outs, ws=ws)

    eager = [t.clone() for t in call()]
    g, out = capture(call)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    hsa.check(ws)
    for a, b in zip(out, eager):
        assert torch.equal(a, b)
