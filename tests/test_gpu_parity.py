"""CUDA path (through the C ABI) against the CPU oracle on identical seeded inputs.

Small cases run the oracle in full; they span several tiles, ragged tails and
the degenerate cases of the method (no visible chunk, fewer visible chunks
than k, exact score ties, every group size). Full-size cases compare sampled
rows and chunks the oracle computes one by one, plus properties that hold at
any size.
"""
import numpy as np
import pytest

import oracle
import synth
from hsa_cases import (TIE_WINDOW, assert_close, bf16_tensor_to_f64, host_inputs, oracle_prefill,
                       to_device_bf16)

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover - collected on CPU only with -m gpu
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2504_16795_gb300 as hsa  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def built():
    hsa.build()
    hsa.load()


def shape_of(w, inner="softmax", weights="softmax"):
    return hsa.Shape(B=w.B, L=w.L, Hq=w.Hq, Hkv=w.Hkv, d=w.d, S=w.S, topk=w.topk, inner=inner, weights=weights)


def run_gpu(w, bits, backward=True, inner="softmax", weights="softmax"):
    shape = shape_of(w, inner, weights)
    q, K, V = (to_device_bf16(bits[n]) for n in ("q", "K", "V"))
    wss = hsa.Workspaces(shape, q.device)
    fwd = hsa.hsa_forward_path(shape, q, K, V, wss)
    out = {k: v for k, v in fwd.items()}
    if backward:
        dO = to_device_bf16(bits["dO"])
        out["dq"], out["dK"], out["dV"] = hsa.hsa_backward_path(shape, q, K, V, fwd, dO, wss)
    torch.cuda.synchronize()
    return out


def check_prefill(w, backward=True, bits=None, inner="softmax", weights="softmax"):
    bits = bits or host_inputs(w, with_dO=backward)
    got = run_gpu(w, bits, backward, inner, weights)
    ref = oracle_prefill(w, bits, backward, inner=inner, weights=weights)
    # chunk summaries: bit-exact fp32 and its bf16 rounding
    kb = got["kbar32"].cpu().numpy()
    assert np.array_equal(kb, ref["kbar32"].astype(np.float32))
    kb16 = got["kbar16"].contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
    assert np.array_equal(kb16, synth.f32_to_bf16(ref["kbar32"].astype(np.float32)))
    # selection: bit-exact indices and scores
    idx = got["idx"].cpu().numpy()
    mismatch = (idx != ref["idx"]).any(axis=-1)
    near_tie = ref["gap"] < TIE_WINDOW
    assert not mismatch.any(), f"{mismatch.sum()} rows differ ({(mismatch & near_tie).sum()} near ties)"
    s_sel = got["s_sel"].cpu().numpy()
    valid = ref["idx"] >= 0
    assert np.array_equal(s_sel[valid], ref["s_sel"][valid].astype(np.float32))
    assert np.isneginf(s_sel[~valid]).all()
    # inverse index: every valid slot listed once under its key, increasing within a key
    off = got["offsets"].cpu().numpy().astype(np.int64)
    ent = got["entries"].cpu().numpy().astype(np.int64)
    flat = ref["idx"].reshape(-1)
    n_valid = int((flat >= 0).sum())
    assert off[0] == 0 and off[-1] == n_valid and (np.diff(off) >= 0).all()
    lst = ent[:n_valid]
    assert np.array_equal(np.sort(lst), np.nonzero(flat >= 0)[0])
    for key in range(len(off) - 1):
        seg = lst[off[key]:off[key + 1]]
        if seg.size:
            assert (np.diff(seg) > 0).all()
            c = key % w.Nc
            assert (flat[seg] == c).all()
    # forward
    assert_close("w", got["w"].cpu().numpy(), ref["w"], max_abs=1e-5, rel=1e-5)
    assert_close("O", bf16_tensor_to_f64(got["O"]), ref["O"])
    if backward:
        assert_close("dq", got["dq"].cpu().numpy(), ref["dq"])
        assert_close("dK", got["dK"].cpu().numpy(), ref["dK"])
        assert_close("dV", got["dV"].cpu().numpy(), ref["dV"])
    return got, ref


SMALL = {
    "tiny (config 1)": synth.WORKLOADS[1],
    "pretrain shape, ragged": synth.WORKLOADS[2].with_(B=2, L=2048 + 37),
    "G16 d128 k16": synth.Workload("g16", 41, B=1, L=2048 + 5, S=64, Hq=16, Hkv=1, d=128, topk=16),
    "G1 d64 k32": synth.Workload("g1", 42, B=2, L=1024 + 63, S=64, Hq=2, Hkv=2, d=64, topk=32),
    "G2 d128 k3": synth.Workload("g2", 43, B=3, L=700, S=64, Hq=8, Hkv=4, d=128, topk=3),
    "G4 d64 k8 offsets": synth.Workload("g4", 44, B=1, L=1536, S=64, Hq=8, Hkv=2, d=64, topk=8,
                                        chunk_offset_sigma=0.5),
}


@pytest.mark.parametrize("name", list(SMALL))
def test_prefill_matches_oracle(name):
    check_prefill(SMALL[name])


@pytest.mark.parametrize("variant", [("softmax1", "softmax"), ("softmax", "stick"), ("softmax1", "stick")])
@pytest.mark.parametrize("name", ["tiny (config 1)", "pretrain shape, ragged", "G16 d128 k16"])
def test_prefill_variants_match_oracle(name, variant):
    # softmax-off-by-one inside chunks (§3.1.2) and stick-breaking chunk weights (§3.1.1)
    inner, weights = variant
    got, ref = check_prefill(SMALL[name], inner=inner, weights=weights)
    keff = (ref["idx"] >= 0).sum(-1)
    if weights == "stick":  # the slots take less than the whole stick
        assert (ref["w"].sum(-1)[keff > 0] < 1.0).all()


@pytest.mark.parametrize("L", [50, 64, 65, 128])
def test_short_sequences(L):
    w = synth.Workload("short", 45, B=2, L=L, S=64, Hq=4, Hkv=2, d=64, topk=4)
    got, ref = check_prefill(w)
    if L <= 64:
        assert (got["idx"].cpu().numpy() == -1).all()
        assert (got["O"].float().cpu().numpy() == 0).all()
        assert (got["dq"].cpu().numpy() == 0).all()
        assert (got["dK"].cpu().numpy() == 0).all() and (got["dV"].cpu().numpy() == 0).all()


def test_exact_score_ties_break_toward_lower_chunk():
    # copy chunk 3 onto chunks 7 and 12: identical summaries give exactly equal
    # scores on both sides; the lower index must rank first
    w = synth.Workload("ties", 46, B=1, L=1024 + 10, S=64, Hq=8, Hkv=1, d=128, topk=2)
    bits = host_inputs(w)
    K = bits["K"]
    for c in (7, 12):
        K[:, c * 64:(c + 1) * 64] = K[:, 3 * 64:4 * 64]
    got, ref = check_prefill(w, bits=bits)
    assert (ref["gap"] == 0).any()


@pytest.mark.parametrize("topk", [8, 16])
def test_selection_many_equal_chunks_takes_the_exact_pass(topk):
    # every complete chunk is a copy of chunk 0: all scores of a row tie, the
    # per-row candidate buffer of the tensor-core selection overflows and the
    # rows go through the exact pass; ties rank the lower chunk index first
    w = synth.Workload("all-equal", 48, B=1, L=64 * 120 + 17, S=64, Hq=8, Hkv=2, d=64, topk=topk)
    bits = host_inputs(w)
    K = bits["K"]
    for c in range(1, w.L // 64):
        K[:, c * 64:(c + 1) * 64] = K[:, 0:64]
    got, ref = check_prefill(w, bits=bits)
    idx = got["idx"].cpu().numpy()
    vis = np.minimum(np.arange(w.L) // 64, w.Nc)
    for t in (200, 64 * 70, w.L - 1):
        keff = min(topk, vis[t])
        assert list(idx[0, t, 0, :keff]) == list(range(keff - 1, -1, -1)), t


def test_backward_is_deterministic():
    w = synth.WORKLOADS[2].with_(B=2, L=2048)
    bits = host_inputs(w)
    a = run_gpu(w, bits)
    b = run_gpu(w, bits)
    for k in ("O", "dq", "dK", "dV"):
        assert torch.equal(a[k], b[k]), k


# ----------------------------------------------------------------------------- full-size workloads

def device_inputs(w, names):
    return {n: synth.device_tensor(w, n) for n in names}


def slice_bits(w, b, g, names):
    """bf16 bits of one (batch, group) slice as a B=1, Hkv=1 problem."""
    G = w.G
    out = {}
    for n in names:
        if n in ("q", "dO"):
            out[n] = synth.host_tensor(w, n, (b, 0, g * G, 0), (b + 1, w.L, (g + 1) * G, w.d))
        else:
            out[n] = synth.host_tensor(w, n, (b, 0, g, 0), (b + 1, w.L, g + 1, w.d))
    return out


@pytest.mark.parametrize("cfg,inner,weights", [(2, "softmax", "softmax"), (3, "softmax", "softmax"),
                                               (3, "softmax1", "stick")])
def test_full_size_sampled(cfg, inner, weights):
    # the variants (softmax-off-by-one inside chunks, stick-breaking chunk
    # weights) at the long-context size, in the bench's launch configuration
    w = synth.WORKLOADS[cfg]
    shape = shape_of(w, inner, weights)
    dev = device_inputs(w, ("q", "K", "V", "dO"))
    wss = hsa.Workspaces(shape, dev["q"].device)
    fwd = hsa.hsa_forward_path(shape, dev["q"], dev["K"], dev["V"], wss)
    dq, dK, dV = hsa.hsa_backward_path(shape, dev["q"], dev["K"], dev["V"], fwd, dev["dO"], wss)
    torch.cuda.synchronize()
    rng = np.random.default_rng(cfg)
    b, g = w.B - 1, w.Hkv - 1
    G = w.G
    bits = slice_bits(w, b, g, ("q", "K", "V", "dO"))
    ws1 = w.with_(B=1, Hq=G, Hkv=1)
    q = synth.bf16_to_f64(bits["q"])
    K = synth.bf16_to_f64(bits["K"])
    V = synth.bf16_to_f64(bits["V"])
    dO = synth.bf16_to_f64(bits["dO"])
    # chunk summaries of the slice, then the whole slice's selection (exact)
    kbar32 = oracle.pool(K, w.S, f32=True)
    assert np.array_equal(fwd["kbar32"][b, :, g].cpu().numpy(), kbar32[0, :, 0].astype(np.float32))
    idx, s_sel, gap = oracle.select(q, kbar32, w.S, w.topk, f32=True)
    got_idx = fwd["idx"][b, :, g].cpu().numpy()
    assert np.array_equal(got_idx, idx[0, :, 0]), f"{(got_idx != idx[0, :, 0]).any(-1).sum()} rows differ"
    # forward on sampled tokens (plus the last one and the first tokens that see a chunk)
    toks = np.unique(np.concatenate([rng.choice(w.L, 384, replace=False), [w.L - 1, 64, 65, 127]]))
    mask = np.zeros((1, w.L), np.uint8)
    mask[0, toks] = 1
    O, wts = oracle.forward(q, K, V, idx, s_sel, w.S, token_mask=mask, inner=inner, weights=weights)
    gotO = bf16_tensor_to_f64(fwd["O"][b, toks, g * G:(g + 1) * G])
    assert_close("O sampled", gotO, O[0, toks])
    # backward: dq on the sampled tokens; dK, dV on sampled chunks, with every
    # token that selected them
    chunks = rng.choice(np.arange(w.Nc // 2, w.Nc - 1), 3, replace=False)
    chunks = np.unique(np.concatenate([chunks, [w.Nc - 1]]))
    sel_any = np.isin(idx[0, :, 0], chunks).any(axis=-1)
    mask2 = mask.copy()
    mask2[0, sel_any] = 1
    kbar64 = oracle.pool(K, w.S)
    ref = oracle.backward(q, K, V, kbar64, idx, s_sel, dO, w.S, token_mask=mask2, inner=inner, weights=weights)
    assert_close("dq sampled", dq[b, toks, g * G:(g + 1) * G].cpu().numpy(), ref["dq"][0, toks])
    for c in chunks:
        rows = slice(c * w.S, (c + 1) * w.S)
        assert_close(f"dK chunk {c}", dK[b, rows, g].cpu().numpy(), ref["dK"][0, rows, 0])
        assert_close(f"dV chunk {c}", dV[b, rows, g].cpu().numpy(), ref["dV"][0, rows, 0])
    assert_close("w sampled", fwd["w"][b, toks, g].cpu().numpy(), wts[0, toks, 0], max_abs=1e-5, rel=1e-5)
    if (inner, weights) != ("softmax", "softmax"):
        return
    # properties at any size: the value gradients add up to dO over tokens with a selection
    keff = (fwd["idx"] >= 0).sum(-1)  # [B, L, Hkv]
    m = (keff > 0).repeat_interleave(G, dim=2).unsqueeze(-1).float()
    want = (dev["dO"].float() * m).view(w.B, w.L, w.Hkv, G, w.d).sum(dim=(1, 3))
    torch.testing.assert_close(dV.sum(dim=1), want, rtol=1e-3, atol=0.5)
    del ws1


def test_full_size_prefill_1m_needles():
    w = synth.WORKLOADS[4]
    shape = shape_of(w)
    dev = device_inputs(w, ("q", "K", "V"))
    wss = hsa.Workspaces(shape, dev["q"].device)
    fwd = hsa.hsa_forward_path(shape, dev["q"], dev["K"], dev["V"], wss)
    torch.cuda.synchronize()
    idx = fwd["idx"][0, :, 0].cpu().numpy()
    # needle property: a needle query selects only needles when >= k are visible, else every visible needle
    needles = np.sort(synth.needle_chunk_ids(w))
    toks = synth.needle_query_tokens(w)
    is_needle = np.zeros(w.Nc + 1, bool)
    is_needle[needles] = True
    nvis_needles = np.searchsorted(needles, toks // w.S)  # needles with index < own chunk
    sel = idx[toks]
    picked = np.where(sel >= 0, is_needle[np.clip(sel, 0, None)], False).sum(axis=1)
    # selections are causal and distinct, so min(k, visible needles) needle picks means
    # "only needles" when >= k are visible and "every visible needle" otherwise
    bad = picked != np.minimum(nvis_needles, w.topk)
    assert not bad.any(), f"{bad.sum()} needle queries miss: first token {toks[bad][0]}"
    # sampled rows against the oracle (exact selection, forward)
    rng = np.random.default_rng(4)
    sample = np.unique(np.concatenate([rng.choice(w.L, 96, replace=False), toks[-32:], [w.L - 1]]))
    Kb = synth.host_tensor(w, "K", (0, 0, 0, 0), w.dims("K"))
    K = synth.bf16_to_f64(Kb)
    kbar32 = oracle.pool(K, w.S, f32=True)
    assert np.array_equal(fwd["kbar32"][0, :, 0].cpu().numpy(), kbar32[0, :, 0].astype(np.float32))
    qb = np.zeros((1, w.L, w.Hq, w.d), np.uint16)
    for t in sample:
        qb[:, t:t + 1] = synth.host_tensor(w, "q", (0, t, 0, 0), (1, t + 1, w.Hq, w.d))
    q = synth.bf16_to_f64(qb)
    mask = np.zeros((1, w.L), np.uint8)
    mask[0, sample] = 1
    ridx, s_sel, gap = oracle.select(q, kbar32, w.S, w.topk, f32=True, token_mask=mask)
    assert np.array_equal(idx[sample], ridx[0, sample, 0])
    V = synth.bf16_to_f64(synth.host_tensor(w, "V", (0, 0, 0, 0), w.dims("V")))
    O, _ = oracle.forward(q, K, V, ridx, s_sel, w.S, token_mask=mask)
    assert_close("O sampled", bf16_tensor_to_f64(fwd["O"][0, sample]), O[0, sample])


# Rows longer than the selection's warm-up: once its bound holds 8k group terms
# (after t_warm tiles of 64 chunks) the kernel collects candidates during its
# one sweep against the bound built so far, and visits only the first t_warm
# tiles again. k = 2 with groups of 32 columns warms up over 8 tiles, k = 12
# (the kernel for k <= 16) over 48; these rows reach 25 and 55 tiles.
@pytest.mark.parametrize("topk,Nc,G,d", [(2, 1600, 2, 64), (12, 3500, 4, 64)])
def test_long_rows_collect_during_the_sweep(topk, Nc, G, d):
    w = synth.Workload("long-rows", 80 + topk, B=1, L=64 * Nc + 13, S=64, Hq=G, Hkv=1, d=d, topk=topk,
                       backward=False)
    shape = shape_of(w)
    dev = device_inputs(w, ("q", "K"))
    kbar32_d, _ = hsa.chunk_pool(shape, dev["K"], want_bf16=False)
    idx, s_sel = hsa.select_topk(shape, dev["q"], kbar32_d)
    torch.cuda.synchronize()
    rng = np.random.default_rng(topk)
    sample = np.unique(np.concatenate([rng.choice(w.L, 256, replace=False), np.arange(w.L - 128, w.L)]))
    K = synth.bf16_to_f64(synth.host_tensor(w, "K", (0, 0, 0, 0), w.dims("K")))
    kbar32 = oracle.pool(K, w.S, f32=True)
    assert np.array_equal(kbar32_d.cpu().numpy(), kbar32.astype(np.float32))
    qb = np.zeros((1, w.L, w.Hq, w.d), np.uint16)
    for t in sample:
        qb[:, t:t + 1] = synth.host_tensor(w, "q", (0, t, 0, 0), (1, t + 1, w.Hq, w.d))
    mask = np.zeros((1, w.L), np.uint8)
    mask[0, sample] = 1
    ridx, rs, _ = oracle.select(synth.bf16_to_f64(qb), kbar32, w.S, w.topk, f32=True, token_mask=mask)
    assert np.array_equal(idx[0, sample].cpu().numpy(), ridx[0, sample])
    assert np.array_equal(s_sel[0, sample].cpu().numpy(), rs[0, sample].astype(np.float32))


def test_full_size_decode_64m_memory():
    w = synth.WORKLOADS[5]
    T, Nc, d = w.L, w.Nc, w.d
    dshape = hsa.DecodeShape(Bq=w.Bq, Hq=w.Hq, Hkv=w.Hkv, d=d, n_chunks=Nc, topk=w.topk)
    pshape = hsa.Shape(B=1, L=T, Hq=w.Hq, Hkv=w.Hkv, d=d, topk=w.topk)
    Kmem = synth.device_tensor(w, "K")
    Vmem = synth.device_tensor(w, "V")
    qd = synth.device_tensor(w, "q")
    kbar32, _ = hsa.chunk_pool(pshape, Kmem.view(1, T, w.Hkv, d), want_bf16=False)
    O, idx, s_sel, wts = hsa.decode(dshape, qd, Kmem, Vmem, kbar32.view(Nc, w.Hkv, d))
    torch.cuda.synchronize()
    idx = idx.cpu().numpy()
    needles = synth.needle_chunk_ids(w)
    for b in range(w.Bq):
        assert needles[b] in idx[b, 0], b
    # oracle: chunk summaries of the whole memory, block by block
    blk = 1 << 20
    kb = np.zeros((Nc, w.Hkv, d))
    for t0 in range(0, T, blk):
        Kbits = synth.host_tensor(w, "K", (0, t0, 0, 0), (1, t0 + blk, w.Hkv, d))
        kb[t0 // w.S:(t0 + blk) // w.S] = oracle.pool(synth.bf16_to_f64(Kbits), w.S, f32=True)[0]
    # sampled summaries bit-exact
    got_kb = kbar32.view(Nc, w.Hkv, d)
    for c in [0, 1, Nc // 2, Nc - 1, int(needles[0])]:
        assert np.array_equal(got_kb[c].cpu().numpy(), kb[c].astype(np.float32))
    q = synth.bf16_to_f64(synth.host_tensor(w, "q", (0, 0, 0, 0), w.dims("q")))[0]
    ridx, rs, gap = oracle.decode_select(q, kb, w.topk, f32=True)
    assert np.array_equal(idx, ridx)
    assert np.array_equal(s_sel.cpu().numpy(), rs.astype(np.float32))
    Ksel = np.zeros((w.Bq, w.Hkv, w.topk, w.S, d))
    Vsel = np.zeros_like(Ksel)
    for b in range(w.Bq):
        for g in range(w.Hkv):
            for j in range(w.topk):
                c = int(ridx[b, g, j])
                Ksel[b, g, j] = synth.bf16_to_f64(synth.host_tensor(w, "K", (0, c * w.S, g, 0),
                                                                    (1, (c + 1) * w.S, g + 1, d)))[0, :, 0]
                Vsel[b, g, j] = synth.bf16_to_f64(synth.host_tensor(w, "V", (0, c * w.S, g, 0),
                                                                    (1, (c + 1) * w.S, g + 1, d)))[0, :, 0]
    rw, rO = oracle.decode_attend(q, Ksel, Vsel, ridx, rs)
    assert_close("decode w", wts.cpu().numpy(), rw, max_abs=1e-5, rel=1e-5)
    assert_close("decode O", bf16_tensor_to_f64(O), rO)


def test_decode_small_memory_against_oracle():
    w = synth.Workload("dec-small", 47, B=1, L=64 * 300, S=64, Hq=8, Hkv=2, d=64, topk=8, backward=False,
                       decode=True, Bq=70, needle_chunks=70)
    T, Nc, d = w.L, w.Nc, w.d
    bits = {n: synth.host_tensor(w, n, (0, 0, 0, 0), w.dims(n)) for n in ("q", "K", "V")}
    qd = to_device_bf16(bits["q"][0])
    Kmem = to_device_bf16(bits["K"][0])
    Vmem = to_device_bf16(bits["V"][0])
    pshape = hsa.Shape(B=1, L=T, Hq=w.Hq, Hkv=w.Hkv, d=d, topk=w.topk)
    kbar32, _ = hsa.chunk_pool(pshape, Kmem.view(1, T, w.Hkv, d), want_bf16=False)
    dshape = hsa.DecodeShape(Bq=w.Bq, Hq=w.Hq, Hkv=w.Hkv, d=d, n_chunks=Nc, topk=w.topk)
    O, idx, s_sel, wts = hsa.decode(dshape, qd, Kmem, Vmem, kbar32.view(Nc, w.Hkv, d))
    torch.cuda.synchronize()
    K = synth.bf16_to_f64(bits["K"])[0]
    V = synth.bf16_to_f64(bits["V"])[0]
    kb = oracle.pool(K[None], w.S, f32=True)[0]
    ref = oracle.decode(synth.bf16_to_f64(bits["q"])[0], K, V, kb, w.S, w.topk, f32=True)
    assert np.array_equal(idx.cpu().numpy(), ref["idx"])
    assert np.array_equal(s_sel.cpu().numpy(), ref["s_sel"].astype(np.float32))
    assert_close("decode w", wts.cpu().numpy(), ref["w"], max_abs=1e-5, rel=1e-5)
    assert_close("decode O", bf16_tensor_to_f64(O), ref["O"])
