"""Edge cases of the selection certificate and of the stick-breaking backward,
CUDA path (through the C ABI) against the CPU oracle.

* Dense near-ties: a cluster of chunks whose summaries all have a large norm
  and differ from one another by one bf16 step in a few coordinates. Their
  exact fp32 scores are distinct but far closer together than the rounding
  bound of the bf16 tensor-core pass, so every one of them is a candidate:
  with a cluster that fits the per-row buffer the rows are certified and
  rescored, with a larger one the buffer overflows and the rows go to the
  exact pass. Indices and scores must equal the fp32 definition bit for bit,
  for prefill selection and for the indexed decode.
* Saturated stick-breaking weights: with a large selection scale the early
  slots take sigmoid(s) = 1 in fp32, so the stick left for later slots is
  below the rounding of the earlier weights; gradients must still meet the
  bars (§3.1.1 "Chunk Weights").
"""
import numpy as np
import pytest

import oracle
import synth
from hsa_cases import assert_close, bf16_tensor_to_f64, host_inputs, to_device_bf16

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover - collected on CPU only with -m gpu
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2504_16795_gb300 as hsa  # noqa: E402

BF16_FOUR = 0x4080  # 4.0 in bf16; one step above it is 4.03125


@pytest.fixture(scope="module", autouse=True)
def built():
    hsa.build()
    hsa.load()


def near_tie_keys(K, cluster, d, seed):
    """Every row of each cluster chunk = 4.0 in every coordinate, plus one bf16 step in n consecutive
    coordinates from a start; each chunk has its own (start, n), so the summaries are distinct (norm about
    4 sqrt(d)). The pairs are assigned to the chunks in a seeded order."""
    order = np.random.default_rng(seed).permutation(len(cluster))
    for j, c in zip(order, cluster):
        row = np.full(d, BF16_FOUR, np.uint16)
        start, n = j % d, 1 + j // d
        row[(start + np.arange(n)) % d] += 1
        K[:, c * 64:(c + 1) * 64, :, :] = row
    return K


def biased_queries(q, bias=1.0):
    """q + bias (one fp32 add per element, rounded to bf16): the group sums point along the cluster."""
    return synth.add_to_bf16(q, np.float32(bias))


def check_spread(kbar, cluster, qhat_rows, scale):
    # the cluster's exact scores are (almost all) distinct and far inside the bf16 pass's rounding bound;
    # the few exact ties (equal coordinates of q̂) must break toward the lower chunk index
    for qh in qhat_rows:
        s = np.array([np.dot(qh, kbar[c]) for c in cluster]) * scale
        assert len(np.unique(s)) >= 0.9 * len(cluster)
        eps = 2.0 ** -7 * 9 / 8 * np.linalg.norm(qh) * np.linalg.norm(kbar[cluster[0]]) * scale
        assert s.max() - s.min() < eps


@pytest.mark.parametrize("d,topk,nclu", [(64, 4, 20), (64, 4, 40), (128, 8, 24), (128, 16, 50), (128, 16, 90)])
def test_selection_is_exact_under_dense_near_ties(d, topk, nclu):
    G = 4
    Nc = 160
    w = synth.Workload("near-ties", 61, B=1, L=64 * Nc + 9, S=64, Hq=G, Hkv=1, d=d, topk=topk)
    bits = host_inputs(w, with_dO=False)
    rng = np.random.default_rng(nclu)
    cluster = np.sort(rng.choice(Nc - 1, nclu, replace=False))
    bits["K"] = near_tie_keys(bits["K"], cluster, d, seed=d + topk)
    bits["q"] = biased_queries(bits["q"])
    shape = hsa.Shape(B=1, L=w.L, Hq=G, Hkv=1, d=d, topk=topk)
    q, K = to_device_bf16(bits["q"]), to_device_bf16(bits["K"])
    kbar32, _ = hsa.chunk_pool(shape, K)
    ws = hsa.new_workspace(hsa.workspace_size(hsa.HSA_OP_SELECT, shape), q.device)
    idx, s_sel = hsa.select_topk(shape, q, kbar32, ws=ws)
    hsa.check(ws)
    q64, K64 = synth.bf16_to_f64(bits["q"]), synth.bf16_to_f64(bits["K"])
    kb = oracle.pool(K64, 64, f32=True)
    ridx, rs, gap = oracle.select(q64, kb, 64, topk, f32=True)
    qhat = q64[0, -1].sum(axis=0)
    check_spread(kb[0, :, 0], cluster, [qhat], shape_scale(G, d))
    got = idx.cpu().numpy()
    bad = (got != ridx).any(-1)
    assert not bad.any(), f"{bad.sum()} rows differ"
    valid = ridx >= 0
    assert np.array_equal(s_sel.cpu().numpy()[valid], rs[valid].astype(np.float32))
    # the last token selects only cluster chunks (they outscore every other chunk)
    assert np.isin(got[0, -1, 0], cluster).all()


def shape_scale(G, d):
    return oracle.default_scales(G, d)[0]


# k = 4 on ranges of 64 chunks takes groups of 8 columns, so a block of at most
# 64 queries scans each row with two threads (one per half of every tile);
# with 150 cluster chunks a range holds about 30, more than one export buffer,
# and the merge scores those ranges exactly.
@pytest.mark.parametrize("topk,nclu", [(8, 20), (8, 60), (4, 20), (4, 150)])
def test_indexed_decode_is_exact_under_dense_near_ties(topk, nclu):
    Nc, d, G = 300, 128, 8
    w = synth.Workload("dec-near-ties", 62, B=1, L=64 * Nc, S=64, Hq=G, Hkv=1, d=d, topk=topk, backward=False,
                       decode=True, Bq=40)
    Kb = synth.host_tensor(w, "K", (0, 0, 0, 0), w.dims("K"))
    rng = np.random.default_rng(nclu)
    cluster = np.sort(rng.choice(Nc, nclu, replace=False))
    Kb = near_tie_keys(Kb, cluster, d, seed=7)
    qb = biased_queries(synth.host_tensor(w, "q", (0, 0, 0, 0), w.dims("q")))[0]
    Kmem = to_device_bf16(Kb[0])
    Vmem = to_device_bf16(synth.host_tensor(w, "V", (0, 0, 0, 0), w.dims("V"))[0])
    qd = to_device_bf16(qb)
    kbar32, _ = hsa.chunk_pool(hsa.Shape(B=1, L=w.L, Hq=G, Hkv=1, d=d, topk=topk), Kmem.view(1, w.L, 1, d),
                               want_bf16=False)
    kbar32 = kbar32.view(Nc, 1, d)
    dshape = hsa.DecodeShape(Bq=w.Bq, Hq=G, Hkv=1, d=d, n_chunks=Nc, topk=topk)
    index = hsa.decode_index(dshape, kbar32)
    ws = hsa.new_workspace(int(hsa.load().hsa_decode_indexed_workspace_size(__import__("ctypes").byref(dshape.c()))),
                           qd.device)
    O, idx, s_sel, wts = hsa.decode_indexed(dshape, qd, Kmem, Vmem, kbar32, index, ws=ws)
    hsa.check(ws)
    K64 = synth.bf16_to_f64(Kb)
    kb = oracle.pool(K64, 64, f32=True)[0]
    q64 = synth.bf16_to_f64(qb)
    check_spread(kb[:, 0], cluster, [q64[b].sum(axis=0) for b in range(3)], shape_scale(G, d))
    ridx, rs, _ = oracle.decode_select(q64, kb, topk, f32=True)
    assert np.array_equal(idx.cpu().numpy(), ridx)
    assert np.array_equal(s_sel.cpu().numpy(), rs.astype(np.float32))
    assert np.isin(ridx, cluster).all()


@pytest.mark.parametrize("scale_sel", [8.0, 16.0])
def test_stick_breaking_backward_with_saturated_scores(scale_sel):
    # scores of tens: sigmoid(s) rounds to 1 in fp32 for the first slots of
    # most rows, so later slots get almost no stick; the gradients still meet
    # the bars and the forward weights stay in [0, 1]
    w = synth.Workload("stick-sat", 63, B=1, L=64 * 24 + 11, S=64, Hq=4, Hkv=1, d=64, topk=6)
    bits = host_inputs(w)
    shape = hsa.Shape(B=1, L=w.L, Hq=4, Hkv=1, d=64, topk=6, scale_sel=scale_sel, weights="stick")
    q, K, V, dO = (to_device_bf16(bits[n]) for n in ("q", "K", "V", "dO"))
    wss = hsa.Workspaces(shape, q.device)
    fwd = hsa.hsa_forward_path(shape, q, K, V, wss)
    dq, dK, dV = hsa.hsa_backward_path(shape, q, K, V, fwd, dO, wss)
    torch.cuda.synchronize()
    wss.check()
    q64, K64, V64, dO64 = (synth.bf16_to_f64(bits[n]) for n in ("q", "K", "V", "dO"))
    kb32 = oracle.pool(K64, 64, f32=True)
    idx, s_sel, _ = oracle.select(q64, kb32, 64, 6, scale_sel=scale_sel, f32=True)
    assert np.array_equal(fwd["idx"].cpu().numpy(), idx)
    # saturation happened: a first-slot score above 17 gives sigmoid = 1 in fp32
    first = s_sel[..., 0][idx[..., 0] >= 0]
    assert (first > 17).mean() > 0.25, first.max()
    O, wts = oracle.forward(q64, K64, V64, idx, s_sel, 64, weights="stick")
    ref = oracle.backward(q64, K64, V64, oracle.pool(K64, 64), idx, s_sel, dO64, 64, scale_sel=scale_sel,
                          weights="stick")
    assert_close("w", fwd["w"].cpu().numpy(), wts, max_abs=1e-5, rel=1e-5)
    assert_close("O", bf16_tensor_to_f64(fwd["O"]), O)
    for name, got in (("dq", dq), ("dK", dK), ("dV", dV)):
        assert_close(name, got.cpu().numpy(), ref[name])
