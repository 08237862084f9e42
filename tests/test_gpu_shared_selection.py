"""Layers that share one selection (§3.1: K, V and the retrieved chunks are
shared across the HSA layers; the selection may use its own q_sel and K^slc):
per-layer hsa_backward_attention accumulates the score gradient, and
hsa_select_backward runs the selection chain once. Checked against the oracle
(attention part with the selection terms switched off, and the selection chain
for the summed ds), and against hsa_backward when the selection inputs are the
attention's own q and K."""
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


def bits_of(w, name, seed_shift, dims):
    ws = w.with_(name=f"{w.name}-{name}", number=w.number + seed_shift) if seed_shift else w
    return synth.host_tensor(ws, name, (0, 0, 0, 0), dims)


CASES = {
    # attention shape (B, L, Hq, Hkv, d, k) and selection shape (Hq_sel, d_sel)
    "G8 d128, selection G2 d64": (synth.Workload("shared", 71, B=2, L=1024 + 37, S=64, Hq=16, Hkv=2, d=128, topk=8),
                                  4, 64),
    "G4 d64, selection G4 d128": (synth.Workload("shared2", 72, B=1, L=1536, S=64, Hq=4, Hkv=1, d=64, topk=4), 4, 128),
}


@pytest.mark.parametrize("weights", ["softmax", "stick"])
@pytest.mark.parametrize("name", list(CASES))
def test_two_layers_sharing_one_selection_match_the_oracle(name, weights):
    w, hq_sel, d_sel = CASES[name]
    B, L, S, k = w.B, w.L, w.S, w.topk
    att = hsa.Shape(B=B, L=L, Hq=w.Hq, Hkv=w.Hkv, d=w.d, S=S, topk=k, weights=weights)
    sel = hsa.Shape(B=B, L=L, Hq=hq_sel, Hkv=w.Hkv, d=d_sel, S=S, topk=k)
    wsel = w.with_(Hq=hq_sel, d=d_sel)
    qs_bits = bits_of(wsel, "q", 100, (B, L, hq_sel, d_sel))
    Ks_bits = bits_of(wsel, "K", 100, (B, L, w.Hkv, d_sel))
    K_bits = bits_of(w, "K", 0, (B, L, w.Hkv, w.d))
    V_bits = bits_of(w, "V", 0, (B, L, w.Hkv, w.d))
    layers = [(bits_of(w, "q", 10 * l, (B, L, w.Hq, w.d)), bits_of(w, "dO", 10 * l, (B, L, w.Hq, w.d))) for l in (0, 1)]

    # GPU: one selection, two layers, the chain once
    q_sel, K_sel = to_device_bf16(qs_bits), to_device_bf16(Ks_bits)
    K, V = to_device_bf16(K_bits), to_device_bf16(V_bits)
    kbar_sel, _ = hsa.chunk_pool(sel, K_sel)
    idx, s_sel = hsa.select_topk(sel, q_sel, kbar_sel)
    offsets, entries = hsa.build_index(sel, idx)
    ds = torch.zeros((B, L, w.Hkv, k), dtype=torch.float32, device=K.device)
    got = []
    for qb, dOb in layers:
        q, dO = to_device_bf16(qb), to_device_bf16(dOb)
        O, wts = hsa.forward(att, q, K, V, idx, s_sel, offsets, entries)
        dq, dK, dV, ds = hsa.backward_attention(att, q, K, V, idx, wts, dO, offsets, entries, ds_accum=ds)
        got.append((O, dq.clone(), dK.clone(), dV.clone()))
    dq_sel, dK_sel = hsa.select_backward(sel, q_sel, kbar_sel, idx, ds, offsets, entries)
    torch.cuda.synchronize()

    # oracle
    qs, Ks = synth.bf16_to_f64(qs_bits), synth.bf16_to_f64(Ks_bits)
    Kf, Vf = synth.bf16_to_f64(K_bits), synth.bf16_to_f64(V_bits)
    kb32 = oracle.pool(Ks, S, f32=True)
    ridx, rs, _ = oracle.select(qs, kb32, S, k, f32=True)
    assert np.array_equal(idx.cpu().numpy(), ridx)
    ds_ref = np.zeros((B, L, w.Hkv, k))
    for (qb, dOb), (O, dq, dK, dV) in zip(layers, got):
        q, dO = synth.bf16_to_f64(qb), synth.bf16_to_f64(dOb)
        O_ref, _ = oracle.forward(q, Kf, Vf, ridx, rs, S, weights=weights)
        g = oracle.backward(q, Kf, Vf, np.zeros((B, L // S, w.Hkv, w.d)), ridx, rs, dO, S, scale_sel=1e-300,
                            weights=weights)
        assert_close("O", bf16_tensor_to_f64(O), O_ref)
        assert_close("dq (attention)", dq.cpu().numpy(), g["dq"])
        assert_close("dK (attention)", dK.cpu().numpy(), g["dK"])
        assert_close("dV", dV.cpu().numpy(), g["dV"])
        ds_ref += g["ds"]
    assert_close("ds (two layers)", ds.cpu().numpy(), ds_ref)
    ref_sel = oracle.select_backward(qs, oracle.pool(Ks, S), ridx, ds_ref, S)
    assert_close("dq_sel", dq_sel.cpu().numpy(), ref_sel["dq"])
    assert_close("dK_sel", dK_sel.cpu().numpy(), ref_sel["dK"])


def close_on_device(name, got, want, max_abs=2e-2, rel=1e-2):
    """The oracle tolerance (max-abs and relative RMS), evaluated on the device for full-size tensors."""
    d = (got.double() - want.double())
    err = d.abs().max().item()
    rr = (d.square().sum() / want.double().square().sum().clamp_min(1e-300)).sqrt().item()
    assert err <= max_abs, f"{name}: max-abs {err:.3e} > {max_abs}"
    assert rr <= rel, f"{name}: rel-RMS {rr:.3e} > {rel}"


@pytest.mark.parametrize("weights", ["softmax", "stick"])
@pytest.mark.parametrize("size", ["pretrain ragged", "long-32k"])
def test_attention_part_plus_selection_chain_is_the_full_backward(size, weights):
    if size == "long-32k":  # the bench's workload, full size
        w = synth.WORKLOADS[3]
        X = {n: synth.device_tensor(w, n) for n in ("q", "K", "V", "dO")}
    else:
        w = synth.WORKLOADS[2].with_(B=1, L=2048 + 40)
        X = {n: to_device_bf16(synth.host_tensor(w, n, (0, 0, 0, 0), w.dims(n))) for n in ("q", "K", "V", "dO")}
    shape = hsa.Shape(B=w.B, L=w.L, Hq=w.Hq, Hkv=w.Hkv, d=w.d, S=w.S, topk=w.topk, weights=weights)
    fwd = hsa.hsa_forward_path(shape, X["q"], X["K"], X["V"])
    dq, dK, dV = hsa.hsa_backward_path(shape, X["q"], X["K"], X["V"], fwd, X["dO"])
    dqa, dKa, dVa, ds = hsa.backward_attention(shape, X["q"], X["K"], X["V"], fwd["idx"], fwd["w"], X["dO"],
                                               fwd["offsets"], fwd["entries"])
    dqs, dKs = hsa.select_backward(shape, X["q"], fwd["kbar32"], fwd["idx"], ds, fwd["offsets"], fwd["entries"])
    torch.cuda.synchronize()
    assert torch.equal(dV, dVa)
    # same mathematics, different rounding: with softmax weights the full backward
    # carries the selection terms through the bf16 dS tile (dS + c_sel ds / S),
    # the split form adds c_sel ds K̄ in fp32; both sit inside the oracle tolerance
    close_on_device("dq", dqa + dqs, dq)
    close_on_device("dK", dKa + dKs, dK)
