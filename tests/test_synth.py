"""The seeded generator follows its published definitions (host side; the
device side is compared bit for bit in test_gpu_synth.py)."""
import numpy as np
import pytest

import synth


def test_splitmix64_known_answers():
    # Reference outputs of SplitMix64 (Steele, Lea & Flood 2014) started in state 1234567.
    want = [6457827717110365317, 3203168211198807973, 9817491932198370423, 4593380528125082431,
            16408922859458223821]
    assert synth.draws_from_state(1234567, 0, 5).tolist() == want
    # counter-based: the n-th output can be drawn on its own
    assert synth.draws_from_state(1234567, 3, 2).tolist() == want[3:]


def test_irwin_hall_moments_and_bounds():
    x = synth.box(42, (1, 1, 1, 1 << 20), (0, 0, 0, 0), (1, 1, 1, 1 << 20), "f32").reshape(-1).astype(np.float64)
    assert abs(x.mean()) < 5e-3
    assert abs(x.var() - 1.0) < 5e-3
    assert np.abs(x).max() <= 6.0
    # values are multiples of 2^-16 (integer sums scaled by a power of two)
    assert np.all(x * 65536 == np.round(x * 65536))
    # the kurtosis of Irwin-Hall(12) is 3 - 1.2/12 = 2.9
    k = ((x - x.mean()) ** 4).mean() / x.var() ** 2
    assert abs(k - 2.9) < 0.02


def test_bf16_rounding_is_round_to_nearest_even():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(0)
    f = (rng.standard_normal(100000) * np.exp(rng.uniform(-20, 20, 100000))).astype(np.float32)
    # exact ties: the dropped half is exactly 0x8000
    ties = (rng.integers(0, 1 << 16, 1000).astype(np.uint32) << 16 | 0x8000).view(np.float32)
    f = np.concatenate([f, ties[np.isfinite(ties)]])
    want = torch.from_numpy(f).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(synth.f32_to_bf16(f), want)
    bits = synth.box(7, (1, 1, 1, 4096), (0, 0, 0, 0), (1, 1, 1, 4096), "bf16").reshape(-1)
    vals = synth.box(7, (1, 1, 1, 4096), (0, 0, 0, 0), (1, 1, 1, 4096), "f32").reshape(-1)
    assert np.array_equal(bits, synth.f32_to_bf16(vals))


def test_box_is_a_slice_of_the_whole_tensor():
    dims = (2, 9, 3, 5)
    full = synth.box(3, dims, (0, 0, 0, 0), dims)
    part = synth.box(3, dims, (1, 2, 1, 1), (2, 7, 3, 4))
    assert np.array_equal(part, full[1:2, 2:7, 1:3, 1:4])


def test_workload_structure_is_planted():
    w = synth.WORKLOADS[2].with_(B=2, L=256)
    K = synth.bf16_to_f64(synth.host_tensor(w, "K", (0, 0, 0, 0), w.dims("K")))
    plain = synth.bf16_to_f64(synth.box(w.seed("K"), w.dims("K"), (0, 0, 0, 0), w.dims("K")))
    off = synth.chunk_offsets(w)
    # each chunk's keys moved by its own offset (up to bf16 rounding)
    moved = (K - plain)[:, : w.Nc * w.S].reshape(2, w.Nc, w.S, w.Hkv, w.d).mean(axis=2)
    assert np.abs(moved - off).max() < 0.05
    w4 = synth.WORKLOADS[4].with_(L=1 << 14)
    ids = synth.needle_chunk_ids(w4)
    assert len(set(ids.tolist())) == w4.needle_chunks and ids.min() >= 1 and ids.max() < w4.Nc
    toks = synth.needle_query_tokens(w4)
    assert 0.1 < toks.size / w4.L < 0.15
    u = synth.needle_direction(w4)
    assert abs(np.linalg.norm(u) - 3.0) < 1e-5
