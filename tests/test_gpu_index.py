"""hsa_build_index against its plain definition: a stable sort of the listed slots by key.

The inverse index (the CSR that replaces the mask M and rank R of §3.1.2) lists, for every key
(b * Hkv + g) * Nc + c, the flat slot ids p = ((b*L + t)*Hkv + g)*topk + j whose idx entry is c,
in increasing p. Slots holding -1 or a chunk id >= Nc are not listed. The selections here are
random (duplicates within a token included), so both the counting sort (Hkv * Nc <= 4096 keys per
batch row) and the radix sort (more keys) are checked bit for bit, with ragged tiles, padding in
the middle of rows and rows that see no chunk at all.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover - collected on CPU only with -m gpu
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2504_16795_gb300 as hsa  # noqa: E402


def random_selection(B, L, Hkv, k, S, seed):
    """idx [B, L, Hkv, k]: visible chunks (c < t // S) drawn with replacement, about 3 % of the
    entries set to -1 and 0.5 % to an id past the last chunk."""
    rng = np.random.default_rng(seed)
    Nc = L // S
    vis = np.minimum(np.arange(L) // S, Nc)[None, :, None, None]
    u = rng.random((B, L, Hkv, k))
    idx = np.where(vis > 0, np.floor(u * np.maximum(vis, 1)).astype(np.int64), -1)
    r = rng.random((B, L, Hkv, k))
    idx = np.where(r < 0.03, -1, idx)
    idx = np.where((r > 0.03) & (r < 0.035), Nc + 1 + (idx & 7), idx)
    return idx.astype(np.int32)


def reference(idx, B, L, Hkv, k, Nc):
    flat = idx.reshape(-1).astype(np.int64)
    p = np.arange(flat.size)
    g = (p // k) % Hkv
    b = p // (k * Hkv * L)
    listed = (flat >= 0) & (flat < Nc)
    key = (b * Hkv + g) * Nc + flat
    order = np.argsort(np.where(listed, key, np.iinfo(np.int64).max), kind="stable")
    n_listed = int(listed.sum())
    offsets = np.searchsorted(np.sort(key[listed]), np.arange(B * Hkv * Nc + 1), side="left")
    return order[:n_listed], offsets, n_listed


CASES = {
    # counting sort: Hkv * Nc <= 4096
    "counting, ragged tiles": (3, 64 * 40 + 17, 2, 4, 64),
    "counting, long rows": (2, 32768, 4, 8, 64),
    "counting, 4096 keys per row": (1, 65536 + 37, 4, 8, 64),
    "counting, one group, k = 16": (2, 8192 + 5, 1, 16, 64),
    # radix sort: more keys per batch row
    "radix, 4104 keys per row": (1, 65536 + 128, 4, 8, 64),
    "radix, 16384 chunks": (1, 1 << 20, 1, 2, 64),
    # no complete chunk: no key at all
    "no chunk": (2, 40, 2, 4, 64),
}


@pytest.mark.parametrize("case", list(CASES))
def test_build_index_is_the_stable_sort_of_the_listed_slots(case):
    B, L, Hkv, k, S = CASES[case]
    Nc = L // S
    idx = random_selection(B, L, Hkv, k, S, seed=hash(case) & 0xFFFF)
    shape = hsa.Shape(B=B, L=L, Hq=Hkv, Hkv=Hkv, d=128, S=S, topk=k)
    d_idx = torch.from_numpy(idx).cuda()
    ws = hsa.new_workspace(hsa.workspace_size(hsa.HSA_OP_INDEX, shape), d_idx.device)
    offsets, entries = hsa.build_index(shape, d_idx, ws=ws)
    torch.cuda.synchronize()
    hsa.check(ws)
    ref_entries, ref_offsets, n_listed = reference(idx, B, L, Hkv, k, Nc)
    got_offsets = offsets.cpu().numpy().astype(np.int64)
    assert np.array_equal(got_offsets, ref_offsets)
    got = entries.cpu().numpy().astype(np.int64)[:n_listed]
    assert np.array_equal(got, ref_entries)
