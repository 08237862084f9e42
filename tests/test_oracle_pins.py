"""Pins for the CPU oracle, independent of the oracle's own code.

Each test checks the oracle against something the paper or the mathematics
fixes (a closed form, a brute-force enumeration on tiny inputs, an invariant,
a special case that reduces to textbook attention, central finite differences)
chosen so that a plausible slip (a dropped term, a wrong sign or index, a
transposed operand, a wrong scale) fails at least one of them.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest

import oracle

RNG = np.random.default_rng(12345)
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def rand(*shape, rng=RNG):
    return rng.standard_normal(shape)


# ----------------------------------------------------------------------------- pool (Appendix A, Eq. 3)

@pytest.mark.parametrize("f32", [False, True])
def test_pool_chunk_size_one_is_identity(f32):
    K = np.round(rand(2, 7, 3, 5) * 64) / 64  # exact in fp32
    kbar = oracle.pool(K, 1, f32=f32)
    assert np.array_equal(kbar, K)


@pytest.mark.parametrize("f32", [False, True])
def test_pool_arithmetic_progression_closed_form(f32):
    B, Nc, S, Hkv, d = 2, 5, 8, 2, 4
    a = np.round(rand(B, Nc, Hkv, d) * 16) / 16
    step = np.round(rand(B, Nc, Hkv, d) * 16) / 16
    s = np.arange(S)[None, None, :, None, None]
    K = (a[:, :, None] + s * step[:, :, None]).reshape(B, Nc * S, Hkv, d)
    L = Nc * S + 3  # ragged tail: the partial chunk is ignored
    K = np.concatenate([K, rand(B, 3, Hkv, d)], axis=1)
    kbar = oracle.pool(K, S, f32=f32)
    assert kbar.shape == (B, Nc, Hkv, d)
    np.testing.assert_array_equal(kbar, a + (S - 1) / 2 * step)
    assert L // S == Nc


def test_pool_is_permutation_invariant_within_a_chunk():
    K = np.round(rand(1, 32, 1, 6) * 8) / 8
    perm = np.concatenate([RNG.permutation(8) + 8 * c for c in range(4)])
    np.testing.assert_array_equal(oracle.pool(K, 8), oracle.pool(K[:, perm], 8))


# ----------------------------------------------------------------------------- selection (Section 3.1)

def brute_force_topk(scores, k):
    """The unique subset T with |T| = min(k, n) such that every member outranks
    every non-member (higher score, or equal score and lower index)."""
    n = len(scores)
    keff = min(k, n)
    found = []
    for T in itertools.combinations(range(n), keff):
        rest = [i for i in range(n) if i not in T]
        if all(scores[i] > scores[r] or (scores[i] == scores[r] and i < r) for i in T for r in rest):
            found.append(T)
    assert len(found) == 1
    return sorted(found[0], reverse=True)


@pytest.mark.parametrize("G,topk", [(1, 2), (2, 3), (4, 1)])
def test_select_matches_subset_enumeration(G, topk):
    B, S, Nc, Hkv, d = 1, 4, 7, 2, 5
    L = Nc * S + 2
    Hq = G * Hkv
    q, K = rand(B, L, Hq, d), rand(B, L, Hkv, d)
    kbar = oracle.pool(K, S)
    scale = 0.37
    idx, s_sel, gap = oracle.select(q, kbar, S, topk, scale_sel=scale)
    # independent score: einsum of the summed group query with the chunk means
    Kc = K[:, : Nc * S].reshape(B, Nc, S, Hkv, d).mean(axis=2)
    qg = q.reshape(B, L, Hkv, G, d).sum(axis=3)
    for b in range(B):
        for t in range(L):
            nvis = min(t // S, Nc)
            for g in range(Hkv):
                sc = [scale * float(qg[b, t, g] @ Kc[b, i, g]) for i in range(nvis)]
                want = brute_force_topk(sc, topk)
                got = [int(x) for x in idx[b, t, g] if x >= 0]
                assert got == want, (t, g)
                assert all(x == -1 for x in idx[b, t, g, len(want):])
                np.testing.assert_allclose(s_sel[b, t, g, : len(want)], [sc[i] for i in want], rtol=1e-12)


def test_select_k_at_least_visible_takes_every_visible_chunk():
    B, L, S, Hq, Hkv, d = 2, 50, 5, 4, 2, 3
    q, K = rand(B, L, Hq, d), rand(B, L, Hkv, d)
    idx, _, gap = oracle.select(q, oracle.pool(K, S), S, topk=L // S + 2)
    for t in range(L):
        nvis = min(t // S, L // S)
        want = list(range(nvis - 1, -1, -1)) + [-1] * (L // S + 2 - nvis)
        assert (idx[:, t] == np.array(want)[None, None, :]).all()
        assert np.isinf(gap[:, t]).all()


def test_select_ties_break_toward_lower_chunk_index():
    # chunks 2 and 3 have identical keys; with k = 2 they tie for the last slot.
    S, d = 2, 4
    means = [1.0, 5.0, 3.0, 3.0, 2.0]
    K = np.zeros((1, S * (len(means) + 1), 1, d))
    for i, m in enumerate(means):
        K[0, i * S:(i + 1) * S, 0, 0] = m
    q = np.zeros((1, K.shape[1], 1, d))
    q[0, -1, 0, 0] = 1.0
    for f32 in (False, True):
        idx, s_sel, gap = oracle.select(q, oracle.pool(K, S, f32=f32), S, topk=2, scale_sel=1.0, f32=f32)
        assert list(idx[0, -1, 0]) == [2, 1]
        assert gap[0, -1, 0] == 0.0


def test_select_is_causal_and_empty_before_first_chunk():
    B, L, S, Hq, Hkv, d = 1, 37, 4, 2, 1, 3
    q, K = rand(B, L, Hq, d), rand(B, L, Hkv, d)
    idx, s_sel, _ = oracle.select(q, oracle.pool(K, S), S, topk=3)
    for t in range(L):
        row = idx[0, t, 0]
        assert (row[row >= 0] < t // S).all()
        if t < S:
            assert (row == -1).all() and np.isneginf(s_sel[0, t, 0]).all()


def test_select_sums_heads_of_a_group():
    # q_1 = -q_0 makes the group query vanish: every score is 0 and the
    # lowest visible indices win the ties.
    B, L, S, d = 1, 40, 4, 6
    q0 = rand(B, L, 1, d)
    q = np.concatenate([q0, -q0], axis=2)
    K = rand(B, L, 1, d) * 3
    idx, s_sel, _ = oracle.select(q, oracle.pool(K, S), S, topk=2)
    for t in range(L):
        nvis = t // S
        want = sorted(range(min(2, nvis)), reverse=True)
        assert list(idx[0, t, 0, : len(want)]) == want
        assert (s_sel[0, t, 0, : len(want)] == 0).all()


def test_select_f32_decision_agrees_with_f64_outside_tie_window():
    B, L, S, Hq, Hkv, d = 1, 512, 16, 4, 2, 32
    q, K = rand(B, L, Hq, d), rand(B, L, Hkv, d)
    i64, _, gap = oracle.select(q, oracle.pool(K, S), S, 4)
    i32, _, _ = oracle.select(q, oracle.pool(K, S, f32=True), S, 4, f32=True)
    differ = (i64 != i32).any(axis=-1)
    assert (gap[differ] < 1e-4).all()


# ----------------------------------------------------------------------------- forward (Section 3.1.1, Algorithm 1)

def run_forward(q, K, V, S, topk, **kw):
    kbar = oracle.pool(K, S)
    idx, s_sel, _ = oracle.select(q, kbar, S, topk, scale_sel=kw.get("scale_sel"))
    O, w = oracle.forward(q, K, V, idx, s_sel, S, scale_attn=kw.get("scale_attn"))
    return idx, s_sel, O, w


def test_forward_constant_values_give_constant_output():
    # Both the per-chunk softmax and the chunk-weight softmax must sum to one.
    B, L, S, Hq, Hkv, d = 2, 70, 8, 4, 2, 5
    q, K = rand(B, L, Hq, d), rand(B, L, Hkv, d)
    V = np.ones((B, L, Hkv, d))
    idx, _, O, w = run_forward(q, K, V, S, 3)
    keff = (idx >= 0).sum(-1)
    has = np.repeat(keff > 0, Hq // Hkv, axis=2)
    np.testing.assert_allclose(O[has], 1.0, atol=1e-14)
    assert (O[~has] == 0).all()
    np.testing.assert_allclose(w.sum(-1)[keff > 0], 1.0, atol=1e-14)
    assert (w[idx < 0] == 0).all()


def test_forward_is_linear_in_values():
    B, L, S, Hq, Hkv, d = 1, 64, 8, 2, 1, 4
    q, K, V = rand(B, L, Hq, d), rand(B, L, Hkv, d), rand(B, L, Hkv, d)
    _, _, O, _ = run_forward(q, K, V, S, 2)
    _, _, O2, _ = run_forward(q, K, 2.0 * V, S, 2)
    np.testing.assert_array_equal(O2, 2.0 * O)


def test_forward_zero_keys_average_the_lowest_chunks():
    # K = 0: every chunk mean and every logit is 0 -> ties pick chunks
    # 0..k_eff-1, w is uniform and each chunk contributes the mean of its values.
    B, L, S, Hq, Hkv, d, k = 1, 45, 5, 3, 1, 4, 3
    q, V = rand(B, L, Hq, d), rand(B, L, Hkv, d)
    K = np.zeros((B, L, Hkv, d))
    idx, _, O, w = run_forward(q, K, V, S, k)
    chunk_means = V[:, : (L // S) * S].reshape(B, L // S, S, Hkv, d).mean(axis=2)
    for t in range(L):
        keff = min(k, t // S)
        want = chunk_means[0, :keff, 0].mean(axis=0) if keff else np.zeros(d)
        for h in range(Hq):
            np.testing.assert_allclose(O[0, t, h], want, atol=1e-13)


def test_forward_chunk_size_one_is_strictly_causal_softmax_attention():
    # S = 1, G = 1, k >= visible: each chunk is one token, the inner softmax is
    # trivial and the chunk weights become causal softmax attention over the
    # previous tokens with scale c_sel.
    B, L, Hq, Hkv, d = 1, 24, 2, 2, 6
    q, K, V = rand(B, L, Hq, d), rand(B, L, Hkv, d), rand(B, L, Hkv, d)
    cs = 0.41
    _, _, O, _ = run_forward(q, K, V, 1, L, scale_sel=cs)
    for t in range(L):
        for h in range(Hq):
            if t == 0:
                assert (O[0, t, h] == 0).all()
                continue
            logits = cs * K[0, :t, h] @ q[0, t, h]
            p = np.exp(logits - logits.max())
            p /= p.sum()
            np.testing.assert_allclose(O[0, t, h], p @ V[0, :t, h], rtol=1e-12, atol=1e-13)


def test_forward_equal_chunk_means_average_textbook_chunk_attention():
    # Each chunk's keys are m + r with the residuals summing to zero, so every
    # chunk mean is m, every score ties, k >= visible gives uniform weights and
    # O_t is the plain mean over visible chunks of softmax(c_att q K_i^T) V_i.
    B, S, Nc, Hq, Hkv, d = 1, 4, 6, 2, 1, 3
    L = S * Nc
    m = rand(d)
    r = rand(Nc, S // 2, d)
    res = np.concatenate([r, -r], axis=1)  # zero sum per chunk
    K = (m[None, None] + res).reshape(1, L, 1, d)
    q, V = rand(B, L, Hq, d), rand(B, L, Hkv, d)
    ca = 0.77
    idx, _, O, w = run_forward(q, K, V, S, Nc, scale_attn=ca)
    for t in range(L):
        nvis = t // S
        for h in range(Hq):
            acc = np.zeros(d)
            for i in range(nvis):
                lg = ca * K[0, i * S:(i + 1) * S, 0] @ q[0, t, h]
                p = np.exp(lg - lg.max())
                p /= p.sum()
                acc += p @ V[0, i * S:(i + 1) * S, 0]
            want = acc / nvis if nvis else acc
            np.testing.assert_allclose(O[0, t, h], want, rtol=1e-10, atol=1e-12)


def test_forward_hand_worked_example():
    with open(os.path.join(GOLDEN, "hand_worked_two_token_chunks.json")) as f:
        g = json.load(f)
    S = g["S"]
    q = np.array(g["q"], float)[None, :, None, :]
    K = np.array(g["K"], float)[None, :, None, :]
    V = np.array(g["V"], float)[None, :, None, :]
    env = {"e": math.e}
    for case in g["cases"]:
        idx, s_sel, O, w = run_forward(q, K, V, S, case["topk"], scale_sel=g["scale_sel"],
                                       scale_attn=g["scale_attn"])
        assert idx[0, :, 0].tolist() == case["idx"]
        if "O" in case:
            want = np.array([[eval(x, {}, env) for x in row] for row in case["O"]])
            np.testing.assert_allclose(O[0, :, 0], want, rtol=1e-14, atol=1e-14)
        if "O_row5" in case:
            want = np.array([eval(x, {}, env) for x in case["O_row5"]])
            np.testing.assert_allclose(O[0, 5, 0], want, rtol=1e-14)


# ----------------------------------------------------------------------------- backward (Algorithms 2-3 + selection chain)

def loss_and_grads(q, K, V, dO, S, topk):
    kbar = oracle.pool(K, S)
    idx, s_sel, _ = oracle.select(q, kbar, S, topk)
    O, w = oracle.forward(q, K, V, idx, s_sel, S)
    g = oracle.backward(q, K, V, kbar, idx, s_sel, dO, S)
    return float((O * dO).sum()), idx, g


def fd_check(name, x, setter, f, grad, n, rng, tol=1e-6):
    flat = x.reshape(-1)
    picks = rng.choice(flat.size, size=min(n, flat.size), replace=False)
    checked = 0
    for p in picks:
        x0 = flat[p]
        h = 1e-5 * max(1.0, abs(x0))
        lp, ip = f(setter(p, x0 + h))
        lm, im = f(setter(p, x0 - h))
        setter(p, x0)
        if not (np.array_equal(ip, im)):
            continue  # the selection moved inside the step: piecewise constant, no gradient
        fd = (lp - lm) / (2 * h)
        an = grad.reshape(-1)[p]
        scale = max(abs(an), 1e-2 * np.abs(grad).max())
        assert abs(fd - an) <= tol * scale, (name, p, fd, an)
        checked += 1
    assert checked >= 0.8 * len(picks)


@pytest.mark.parametrize("topk", [2, 1])
def test_backward_matches_central_finite_differences(topk):
    rng = np.random.default_rng(7 + topk)
    B, L, S, Hq, Hkv, d = 1, 256, 16, 2, 1, 8
    q, K, V, dO = (rng.standard_normal(s) for s in [(B, L, Hq, d), (B, L, Hkv, d), (B, L, Hkv, d), (B, L, Hq, d)])
    _, idx0, g = loss_and_grads(q, K, V, dO, S, topk)
    if topk == 1:
        assert np.abs(g["ds"]).max() == 0.0  # one chunk: w = 1, no score gradient
    else:
        assert np.abs(g["ds"]).max() > 1e-3

    for name, arr in (("q", q), ("K", K), ("V", V)):
        flat = arr.reshape(-1)

        def setter(p, v, flat=flat):
            flat[p] = v
            return None

        def f(_):
            kbar = oracle.pool(K, S)
            idx, s_sel, _ = oracle.select(q, kbar, S, topk)
            O, _w = oracle.forward(q, K, V, idx, s_sel, S)
            return float((O * dO).sum()), idx

        fd_check(name, arr, setter, f, g["d" + name], 60, rng)


def test_backward_invariants():
    rng = np.random.default_rng(3)
    B, L, S, Hq, Hkv, d, k = 2, 130, 8, 4, 2, 6, 3
    q, K, V, dO = (rng.standard_normal(s) for s in [(B, L, Hq, d), (B, L, Hkv, d), (B, L, Hkv, d), (B, L, Hq, d)])
    _, idx, g = loss_and_grads(q, K, V, dO, S, k)
    # softmax-gradient rows sum to zero
    np.testing.assert_allclose(g["ds"].sum(-1), 0.0, atol=1e-12)
    # inner softmax-gradient rows sum to zero, so a chunk's key gradients sum to dK̄
    Nc = L // S
    chunk_sum = g["dK"][:, : Nc * S].reshape(B, Nc, S, Hkv, d).sum(axis=2)
    np.testing.assert_allclose(chunk_sum, g["dkbar"], atol=1e-11)
    # P rows and w both sum to one: the values' gradients add up to dO over tokens with a selection
    keff = (idx >= 0).sum(-1)  # [B, L, Hkv]
    G = Hq // Hkv
    mask = np.repeat(keff > 0, G, axis=2)[..., None]
    want = (dO * mask).reshape(B, L, Hkv, G, d).sum(axis=(1, 3))
    np.testing.assert_allclose(g["dV"].sum(axis=1), want, atol=1e-11)
    # the partial trailing chunk and the first token chunk never receive gradient through selection
    assert (g["dK"][:, Nc * S:] == 0).all() and (g["dV"][:, Nc * S:] == 0).all()
    assert (g["dq"][:, :S] == 0).all()


# ----------------------------------------------------------------------------- variants: stick-breaking weights
# (§3.1.1 "Chunk Weights") and softmax-off-by-one inside a chunk (§3.1.2 "Kernel Design")

def sigmoid(x):
    return 0.5 * (1.0 + np.tanh(0.5 * x))


def test_stick_breaking_leaves_the_product_of_the_refusals():
    # the slots share a unit stick: what they take together is 1 - prod(1 - sigmoid(s))
    rng = np.random.default_rng(21)
    B, L, S, Hq, Hkv, d, k = 1, 96, 8, 2, 1, 4, 4
    q, K = rng.standard_normal((B, L, Hq, d)), rng.standard_normal((B, L, Hkv, d))
    V = np.ones((B, L, Hkv, d))
    kbar = oracle.pool(K, S)
    idx, s_sel, _ = oracle.select(q, kbar, S, k)
    O, w = oracle.forward(q, K, V, idx, s_sel, S, weights="stick")
    keff = (idx >= 0).sum(-1)
    for t in range(L):
        n = keff[0, t, 0]
        left = np.prod([1.0 - sigmoid(x) for x in s_sel[0, t, 0, :n]]) if n else 1.0
        np.testing.assert_allclose(w[0, t, 0].sum(), 1.0 - left, atol=1e-14)
        np.testing.assert_allclose(O[0, t], 1.0 - left, atol=1e-13)  # constant values: O = taken share
        assert (w[0, t, 0, n:] == 0).all()


def test_stick_breaking_with_equal_scores_is_geometric_from_the_latest_chunk():
    # equal selection scores (identical chunk means): slot j (j-th latest chunk)
    # takes b (1 - b)^j with b = sigmoid(s)
    B, S, Nc, Hq, Hkv, d, k = 1, 4, 8, 1, 1, 3, 5
    L = S * Nc
    m = np.array([0.3, -0.2, 0.5])
    r = RNG.standard_normal((Nc, S // 2, d))
    K = (m[None, None] + np.concatenate([r, -r], axis=1)).reshape(1, L, 1, d)
    q, V = RNG.standard_normal((B, L, Hq, d)), RNG.standard_normal((B, L, Hkv, d))
    kbar = oracle.pool(K, S)
    idx, s_sel, _ = oracle.select(q, kbar, S, k)
    _, w = oracle.forward(q, K, V, idx, s_sel, S, weights="stick")
    for t in range(S, L):
        n = min(k, t // S)
        b = sigmoid(s_sel[0, t, 0, 0])
        np.testing.assert_allclose(w[0, t, 0, :n], b * (1.0 - b) ** np.arange(n), rtol=1e-12)
        assert (np.diff(idx[0, t, 0, :n]) < 0).all()  # slot order: the latest chunk first


def test_softmax_off_by_one_on_single_token_chunks_is_a_sigmoid_gate():
    # S = 1: each chunk is one token, the inner softmax-off-by-one is sigmoid(c_att q·k)
    rng = np.random.default_rng(5)
    B, L, Hq, Hkv, d = 1, 20, 2, 1, 5
    q, K, V = rng.standard_normal((B, L, Hq, d)), rng.standard_normal((B, L, Hkv, d)), rng.standard_normal((B, L, Hkv, d))
    ca = 0.6
    kbar = oracle.pool(K, 1)
    idx, s_sel, _ = oracle.select(q, kbar, 1, L)
    O, w = oracle.forward(q, K, V, idx, s_sel, 1, scale_attn=ca, inner="softmax1")
    for t in range(1, L):
        for h in range(Hq):
            acc = np.zeros(d)
            for j, c in enumerate(idx[0, t, 0]):
                if c < 0:
                    break
                acc += w[0, t, 0, j] * sigmoid(ca * q[0, t, h] @ K[0, c, 0]) * V[0, c, 0]
            np.testing.assert_allclose(O[0, t, h], acc, rtol=1e-12, atol=1e-14)


def test_softmax_off_by_one_with_constant_values_keeps_z_over_one_plus_z():
    rng = np.random.default_rng(9)
    B, L, S, Hq, Hkv, d, k = 1, 48, 8, 2, 1, 4, 3
    q, K = rng.standard_normal((B, L, Hq, d)), 2.0 * rng.standard_normal((B, L, Hkv, d))
    V = np.ones((B, L, Hkv, d))
    ca = 0.9
    kbar = oracle.pool(K, S)
    idx, s_sel, _ = oracle.select(q, kbar, S, k)
    O, w = oracle.forward(q, K, V, idx, s_sel, S, scale_attn=ca, inner="softmax1")
    for t in range(S, L):
        for h in range(Hq):
            want = 0.0
            for j, c in enumerate(idx[0, t, 0]):
                if c < 0:
                    break
                z = np.exp(ca * K[0, c * S:(c + 1) * S, 0] @ q[0, t, h]).sum()
                want += w[0, t, 0, j] * z / (1.0 + z)
            np.testing.assert_allclose(O[0, t, h], want, rtol=1e-12)


@pytest.mark.parametrize("inner,weights,topk", [("softmax1", "softmax", 2), ("softmax", "stick", 3),
                                                ("softmax1", "stick", 2), ("softmax", "stick", 1)])
def test_variant_backward_matches_central_finite_differences(inner, weights, topk):
    rng = np.random.default_rng(11 + topk)
    B, L, S, Hq, Hkv, d = 1, 192, 16, 2, 1, 8
    q, K, V, dO = (rng.standard_normal(s) for s in [(B, L, Hq, d), (B, L, Hkv, d), (B, L, Hkv, d), (B, L, Hq, d)])
    kbar = oracle.pool(K, S)
    idx0, s0, _ = oracle.select(q, kbar, S, topk)
    g = oracle.backward(q, K, V, kbar, idx0, s0, dO, S, inner=inner, weights=weights)
    if weights == "stick":
        assert np.abs(g["ds"]).max() > 1e-3  # even one chunk: w = sigmoid(s) depends on its score

    for name, arr in (("q", q), ("K", K), ("V", V)):
        flat = arr.reshape(-1)

        def setter(p, v, flat=flat):
            flat[p] = v
            return None

        def f(_):
            kb = oracle.pool(K, S)
            idx, s_sel, _ = oracle.select(q, kb, S, topk)
            O, _w = oracle.forward(q, K, V, idx, s_sel, S, inner=inner, weights=weights)
            return float((O * dO).sum()), idx

        fd_check(name, arr, setter, f, g["d" + name], 50, rng)


# ----------------------------------------------------------------------------- the selection chain on its own
# (layers that share one selection add their score gradients, then the chain runs once)

def test_selection_backward_is_the_gradient_of_the_scores_against_fixed_weights():
    # loss = sum ds * s_sel(q, K) with ds fixed: its gradient is exactly the selection chain
    rng = np.random.default_rng(17)
    B, L, S, Hq, Hkv, d, k = 1, 160, 16, 4, 2, 6, 3
    q, K = rng.standard_normal((B, L, Hq, d)), rng.standard_normal((B, L, Hkv, d))
    kbar = oracle.pool(K, S)
    idx0, _, _ = oracle.select(q, kbar, S, k)
    ds = rng.standard_normal(idx0.shape) * (idx0 >= 0)
    g = oracle.select_backward(q, kbar, idx0, ds, S)

    for name, arr in (("q", q), ("K", K)):
        flat = arr.reshape(-1)

        def setter(p, v, flat=flat):
            flat[p] = v
            return None

        def f(_):
            kb = oracle.pool(K, S)
            idx, s_sel, _ = oracle.select(q, kb, S, k)
            return float((np.where(idx >= 0, s_sel, 0.0) * ds).sum()), idx

        fd_check(name, arr, setter, f, g["d" + name], 60, rng)


def test_full_backward_is_attention_part_plus_selection_chain():
    rng = np.random.default_rng(19)
    B, L, S, Hq, Hkv, d, k = 2, 130, 8, 4, 2, 6, 3
    q, K, V, dO = (rng.standard_normal(s) for s in [(B, L, Hq, d), (B, L, Hkv, d), (B, L, Hkv, d), (B, L, Hq, d)])
    kbar = oracle.pool(K, S)
    idx, s_sel, _ = oracle.select(q, kbar, S, k)
    full = oracle.backward(q, K, V, kbar, idx, s_sel, dO, S)
    att = oracle.backward(q, K, V, kbar, idx, s_sel, dO, S, scale_sel=1e-300)  # selection terms vanish
    sel = oracle.select_backward(q, kbar, idx, full["ds"], S)
    np.testing.assert_allclose(att["ds"], full["ds"], atol=1e-14)
    np.testing.assert_allclose(att["dq"] + sel["dq"], full["dq"], atol=1e-12)
    np.testing.assert_allclose(att["dK"] + sel["dK"], full["dK"], atol=1e-12)
    np.testing.assert_allclose(sel["dkbar"], full["dkbar"], atol=1e-12)


# ----------------------------------------------------------------------------- decode (Section 3.2, Inference)

def test_decode_equals_the_forward_row_after_the_memory():
    rng = np.random.default_rng(11)
    S, Nc, Hq, Hkv, d, k = 4, 9, 4, 2, 5, 3
    T = S * Nc
    Kmem, Vmem = rng.standard_normal((T, Hkv, d)), rng.standard_normal((T, Hkv, d))
    qd = rng.standard_normal((3, Hq, d))
    kbar = oracle.pool(Kmem[None], S)[0]
    dec = oracle.decode(qd, Kmem, Vmem, kbar, S, k)
    for b in range(3):
        # the same query as token T of a sequence whose first T tokens are the memory
        q = np.zeros((1, T + 1, Hq, d))
        q[0, T] = qd[b]
        K = np.concatenate([Kmem, rng.standard_normal((1, Hkv, d))])[None]
        V = np.concatenate([Vmem, rng.standard_normal((1, Hkv, d))])[None]
        idx, s_sel, O, w = run_forward(q, K, V, S, k)
        assert (idx[0, T] == dec["idx"][b]).all()
        np.testing.assert_allclose(O[0, T], dec["O"][b], rtol=1e-12, atol=1e-14)


def test_decode_finds_a_planted_needle_chunk():
    rng = np.random.default_rng(5)
    S, Nc, Hq, Hkv, d, k = 8, 300, 4, 1, 16, 4
    Kmem = rng.standard_normal((S * Nc, Hkv, d))
    u = rng.standard_normal(d)
    u *= 3 / np.linalg.norm(u)
    needle = 137
    Kmem[needle * S:(needle + 1) * S, 0] += u
    q = rng.standard_normal((1, Hq, d)) + u
    kbar = oracle.pool(Kmem[None], S)[0]
    for f32 in (False, True):
        idx, _, _ = oracle.decode_select(q, kbar, k, f32=f32)
        assert needle in idx[0, 0]
