"""The C ABI loads, exports everything include/*.h declares, and validates
arguments before any launch (these calls never reach the GPU)."""
import ctypes
import os
import re

import pytest

import paper_2504_16795_gb300 as hsa
import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

OK, INVALID, UNSUPPORTED, WORKSPACE, CUDA, TIMEOUT, BOUNDS = 0, 1, 2, 3, 4, 5, 6


def declared(header):
    text = open(header).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b((?:hsa|synth_dev)_\w+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    hsa.build()
    return hsa.load()


def test_library_exports_every_declared_entry_point(lib):
    names = declared(os.path.join(ROOT, "include", "hsa.h"))
    assert {"hsa_chunk_pool", "hsa_select_topk", "hsa_build_index", "hsa_forward", "hsa_backward",
            "hsa_decode"} <= set(names)
    for n in names:
        assert hasattr(lib, n), n


def test_synth_device_library_exports_its_header():
    dev = ctypes.CDLL(synth.build_device())
    for n in declared(os.path.join(ROOT, "synth", "synth.h")):
        assert hasattr(dev, n), n


def test_status_strings(lib):
    for code in (OK, INVALID, UNSUPPORTED, WORKSPACE, CUDA, TIMEOUT, BOUNDS):
        assert hsa.status_string(code).startswith("HSA_")
    assert hsa.status_string(BOUNDS).startswith("HSA_ERR_BOUNDS")


def test_debug_bounds_library_exports_every_declared_entry_point():
    # the HSA_DEBUG_BOUNDS build: the same entry points, index checks inside
    from paper_2504_16795_gb300.build import build as build_hsa

    dbg = ctypes.CDLL(build_hsa(debug_bounds=True))
    for n in declared(os.path.join(ROOT, "include", "hsa.h")):
        assert hasattr(dbg, n), n


def shape(**kw):
    base = dict(B=1, L=1024, Hq=8, Hkv=1, d=128, S=64, topk=8)
    base.update(kw)
    return hsa.Shape(**base)


FAKE = 1 << 20  # an aligned address that is never dereferenced: every call below fails validation first


def call_forward(lib, s, ws_bytes=None, **ptrs):
    p = dict(q=FAKE, K=FAKE, V=FAKE, idx=FAKE, s_sel=FAKE, off=FAKE, ent=FAKE, O=FAKE, w=FAKE, ws=FAKE)
    p.update(ptrs)
    need = hsa.workspace_size(hsa.HSA_OP_FORWARD, s)
    c = s.c()
    vp = ctypes.c_void_p
    return lib.hsa_forward(ctypes.byref(c), vp(p["q"]), vp(p["K"]), vp(p["V"]), vp(p["idx"]), vp(p["s_sel"]),
                           vp(p["off"]), vp(p["ent"]), vp(p["O"]), vp(p["w"]), vp(p["ws"]),
                           need if ws_bytes is None else ws_bytes, None)


@pytest.mark.parametrize("kw,code", [
    (dict(d=96), UNSUPPORTED),
    (dict(d=256), UNSUPPORTED),
    (dict(Hq=12, Hkv=4), UNSUPPORTED),   # G = 3
    (dict(Hq=64, Hkv=2), UNSUPPORTED),   # G = 32
    (dict(S=32), UNSUPPORTED),
    (dict(topk=33), UNSUPPORTED),
    (dict(Hq=6, Hkv=4), INVALID),        # not a multiple
    (dict(topk=0), INVALID),
    (dict(L=-1), INVALID),
    (dict(B=1 << 20, L=1 << 20), UNSUPPORTED),  # slot count overflows int32
])
def test_shape_validation(lib, kw, code):
    assert call_forward(lib, shape(**kw), ws_bytes=0) == code


def test_unknown_variant_flags_are_unsupported(lib):
    c = shape().c()
    c.flags = 4
    vp = ctypes.c_void_p
    assert lib.hsa_forward(ctypes.byref(c), *[vp(FAKE)] * 10, 1 << 30, None) == UNSUPPORTED
    d = hsa.DecodeShape(Bq=4, Hq=8, Hkv=1, d=128, n_chunks=100).c()
    d.flags = 8
    assert lib.hsa_decode(ctypes.byref(d), *[vp(FAKE)] * 9, 1 << 30, None) == UNSUPPORTED
    with pytest.raises(ValueError):
        shape(weights="uniform").flags


def test_stick_breaking_backward_needs_its_extra_workspace(lib):
    base = hsa.workspace_size(hsa.HSA_OP_BACKWARD, shape())
    stick = hsa.workspace_size(hsa.HSA_OP_BACKWARD, shape(weights="stick"))
    s = shape()
    rows, slots = s.B * s.L * s.Hkv, s.B * s.L * s.Hkv * s.topk
    # stick-breaking: no Δ; dw and ds per slot and the fp32 q̂ rows instead
    assert stick == base - rows * 4 + 2 * slots * 4 + rows * s.d * 4
    att = hsa.workspace_size(hsa.HSA_OP_BACKWARD_ATTENTION, s)
    assert att == base - rows * 4 + slots * 4  # dq partials and dw
    assert hsa.workspace_size(hsa.HSA_OP_SELECT_BACKWARD, s) == hsa.status_bytes() + rows * s.d * 4


def test_null_and_misaligned_pointers_are_rejected(lib):
    s = shape()
    assert call_forward(lib, s, q=0) == INVALID
    assert call_forward(lib, s, K=FAKE + 8) == INVALID
    assert call_forward(lib, s, O=FAKE + 2) == INVALID


def test_short_workspace_is_rejected(lib):
    s = shape()
    need = hsa.workspace_size(hsa.HSA_OP_FORWARD, s)
    assert need > 0
    assert call_forward(lib, s, ws_bytes=need - 1) == WORKSPACE
    assert call_forward(lib, s, ws=0) == WORKSPACE
    need = hsa.workspace_size(hsa.HSA_OP_SELECT, s)
    assert need > 0
    c = s.c()
    vp = ctypes.c_void_p
    assert lib.hsa_select_topk(ctypes.byref(c), *[vp(FAKE)] * 5, need - 1, None) == WORKSPACE


def test_empty_problems_succeed_without_launching(lib):
    assert call_forward(lib, shape(B=0), q=0, K=0, V=0) == OK
    assert call_forward(lib, shape(L=0), q=0, K=0, V=0) == OK
    d = hsa.DecodeShape(Bq=0, Hq=8, Hkv=1, d=128, n_chunks=10)
    c = d.c()
    vp = ctypes.c_void_p
    assert lib.hsa_decode(ctypes.byref(c), *[vp(0)] * 9, 0, None) == OK


def test_decode_validation(lib):
    vp = ctypes.c_void_p
    for kw, code in [(dict(d=80), UNSUPPORTED), (dict(n_chunks=-1), INVALID), (dict(topk=40), UNSUPPORTED)]:
        base = dict(Bq=4, Hq=8, Hkv=1, d=128, n_chunks=100)
        base.update(kw)
        c = hsa.DecodeShape(**base).c()
        assert lib.hsa_decode(ctypes.byref(c), *[vp(FAKE)] * 9, 1 << 30, None) == code
    c = hsa.DecodeShape(Bq=4, Hq=8, Hkv=1, d=128, n_chunks=100).c()
    assert lib.hsa_decode(ctypes.byref(c), *[vp(FAKE)] * 9, 16, None) == WORKSPACE


def test_decode_noalloc_rejects_shapes_beyond_its_scratch(lib):
    vp = ctypes.c_void_p
    limit = 8 << 20
    big = hsa.DecodeShape(Bq=1024, Hq=8, Hkv=1, d=128, n_chunks=1 << 20)
    assert hsa.decode_workspace_size(big) > limit
    c = big.c()
    assert lib.hsa_decode_noalloc(ctypes.byref(c), *[vp(FAKE)] * 8, None) == WORKSPACE
    # 64 queries over a 2^26-token memory fit
    assert hsa.decode_workspace_size(hsa.DecodeShape(Bq=64, Hq=8, Hkv=1, d=128, n_chunks=1 << 20)) <= limit
    c = hsa.DecodeShape(Bq=0, Hq=8, Hkv=1, d=128, n_chunks=10).c()
    assert lib.hsa_decode_noalloc(ctypes.byref(c), *[vp(0)] * 8, None) == OK
    c = hsa.DecodeShape(Bq=4, Hq=8, Hkv=1, d=80, n_chunks=10).c()
    assert lib.hsa_decode_noalloc(ctypes.byref(c), *[vp(FAKE)] * 8, None) == UNSUPPORTED
    c = hsa.DecodeShape(Bq=4, Hq=8, Hkv=1, d=128, n_chunks=10).c()
    assert lib.hsa_decode_noalloc(ctypes.byref(c), *[vp(FAKE + 8)] * 8, None) == INVALID


def test_decode_index_sizes_and_fallback(lib):
    vp = ctypes.c_void_p
    s = hsa.DecodeShape(Bq=64, Hq=8, Hkv=1, d=128, n_chunks=1 << 20, topk=8)
    c = s.c()
    # bf16 summaries + one fp32 norm per chunk + one max per 64 chunks
    assert lib.hsa_decode_index_size(ctypes.byref(c)) >= (1 << 20) * (128 * 2 + 4)
    assert lib.hsa_decode_indexed_workspace_size(ctypes.byref(c)) > 0
    big_k = hsa.DecodeShape(Bq=64, Hq=8, Hkv=1, d=128, n_chunks=1 << 20, topk=20).c()
    assert lib.hsa_decode_index_size(ctypes.byref(big_k)) == 0
    assert lib.hsa_decode_index(ctypes.byref(big_k), vp(FAKE), vp(FAKE), 0, None) == UNSUPPORTED
    assert lib.hsa_decode_index(ctypes.byref(c), vp(FAKE), vp(FAKE), 16, None) == WORKSPACE
    # a missing index is an invalid argument (checked before any launch)
    assert lib.hsa_decode_indexed(ctypes.byref(c), *[vp(FAKE)] * 4, vp(0), *[vp(FAKE)] * 5, 1 << 40, None) == INVALID


def test_growing_memory_capacity_and_append_validation(lib):
    vp, ll = ctypes.c_void_p, ctypes.c_longlong
    # the index of a growing memory is laid out for its capacity, whatever it holds now
    grown = hsa.DecodeShape(Bq=8, Hq=8, Hkv=2, d=64, n_chunks=1000).c()
    empty = hsa.DecodeShape(Bq=8, Hq=8, Hkv=2, d=64, n_chunks=0, capacity_chunks=1000).c()
    part = hsa.DecodeShape(Bq=8, Hq=8, Hkv=2, d=64, n_chunks=371, capacity_chunks=1000).c()
    n = lib.hsa_decode_index_size(ctypes.byref(grown))
    assert n > 0 and lib.hsa_decode_index_size(ctypes.byref(empty)) == n == lib.hsa_decode_index_size(
        ctypes.byref(part))
    assert lib.hsa_decode_index(ctypes.byref(empty), vp(FAKE), vp(FAKE), n - 16, None) == WORKSPACE
    # capacity below the chunks present
    bad = hsa.DecodeShape(Bq=8, Hq=8, Hkv=2, d=64, n_chunks=10, capacity_chunks=9).c()
    assert lib.hsa_decode_workspace_size(ctypes.byref(bad)) == 0
    assert lib.hsa_decode_index(ctypes.byref(bad), vp(FAKE), vp(FAKE), 1 << 30, None) == INVALID
    ptrs = [vp(FAKE)] * 5

    def append(shape, n_tokens, n_new, index=None, nbytes=0, p=ptrs):
        return lib.hsa_memory_append(ctypes.byref(shape), ll(n_tokens), ll(n_new), *p, index, nbytes, None)

    assert append(empty, 0, 0) == OK
    assert append(empty, 1000 * 64, 0) == OK
    assert append(empty, 1000 * 64 - 5, 6) == INVALID  # past the capacity
    assert append(empty, -1, 4) == INVALID
    assert append(empty, 0, -4) == INVALID
    assert append(empty, 0, 64, p=[vp(FAKE), vp(0), vp(FAKE), vp(FAKE), vp(FAKE)]) == INVALID
    assert append(empty, 0, 64, p=[vp(FAKE)] * 4 + [vp(FAKE + 4)]) == INVALID
    assert append(empty, 0, 64, vp(FAKE), n - 1) == WORKSPACE
    assert append(empty, 0, 64, vp(FAKE + 8), n) == WORKSPACE
    big_k = hsa.DecodeShape(Bq=8, Hq=8, Hkv=2, d=64, n_chunks=0, capacity_chunks=1000, topk=20).c()
    assert lib.hsa_decode_index_size(ctypes.byref(big_k)) == 0
    assert append(big_k, 0, 64, vp(FAKE), 1 << 30) == UNSUPPORTED
    odd = hsa.DecodeShape(Bq=8, Hq=8, Hkv=2, d=96, n_chunks=0, capacity_chunks=1000).c()
    assert append(odd, 0, 64) == UNSUPPORTED


def test_workspace_sizes_scale_with_the_problem(lib):
    s = shape(B=2, L=32768, Hq=32, Hkv=4)
    slots = 2 * 32768 * 4 * 8
    # selection on the tensor cores keeps q̂ (bf16 and fp32) per (b, g, t) row
    assert hsa.workspace_size(hsa.HSA_OP_SELECT, s) >= 2 * 32768 * 4 * 128 * 6
    # the CUDA-core selection (k > 16) needs only the status header
    assert hsa.workspace_size(hsa.HSA_OP_SELECT, shape(B=2, L=32768, Hq=32, Hkv=4, topk=24)) == hsa.status_bytes()
    # the forward keeps one bf16 partial per slot and head, and the list of slot-list segments
    assert hsa.workspace_size(hsa.HSA_OP_FORWARD, s) >= hsa.status_bytes() + slots * 8 * 128 * 2
    assert hsa.workspace_size(hsa.HSA_OP_BACKWARD, s) >= slots * 8 * 128 * 2
    # the index: with Hkv * Nc <= 4096 keys per batch row, one count per (key, tile of 8192 slots)
    n_tiles = -(-32768 // (8192 // (4 * 8)))
    assert hsa.workspace_size(hsa.HSA_OP_INDEX, s) >= 2 * 4 * 512 * n_tiles * 4
    # with more keys per row, the radix sort's two key and value buffers
    long_row = shape(B=1, L=1 << 20, Hq=16, Hkv=1, topk=16)
    assert hsa.workspace_size(hsa.HSA_OP_INDEX, long_row) >= (1 << 20) * 16 * 16
    assert hsa.workspace_size(hsa.HSA_OP_FORWARD, shape(d=96)) == 0


def test_every_workspace_starts_with_the_status_header(lib):
    assert hsa.status_bytes() == 256
    s = shape()
    for op in (hsa.HSA_OP_SELECT, hsa.HSA_OP_INDEX, hsa.HSA_OP_FORWARD, hsa.HSA_OP_BACKWARD,
               hsa.HSA_OP_BACKWARD_ATTENTION, hsa.HSA_OP_SELECT_BACKWARD):
        assert hsa.workspace_size(op, s) > hsa.status_bytes(), op
        assert hsa.workspace_size(op, shape(B=0)) == 0, op  # an empty problem takes none
    d = hsa.DecodeShape(Bq=4, Hq=8, Hkv=1, d=128, n_chunks=100)
    assert hsa.decode_workspace_size(d) > hsa.status_bytes()
    c = d.c()
    assert lib.hsa_decode_indexed_workspace_size(ctypes.byref(c)) > hsa.status_bytes()
    # a workspace of the header alone is not enough for a call that needs scratch
    assert call_forward(lib, s, ws_bytes=hsa.status_bytes()) == WORKSPACE


def test_check_and_selftest_validate_their_workspace(lib):
    vp = ctypes.c_void_p
    n = hsa.status_bytes()
    assert lib.hsa_check(vp(0), n, None) == INVALID
    assert lib.hsa_check(vp(FAKE + 4), n, None) == INVALID
    assert lib.hsa_check(vp(FAKE), n - 1, None) == INVALID
    before = lib.hsa_kernel_launches()
    assert lib.hsa_selftest_wait_timeout(1000, vp(0), n, None) == WORKSPACE
    assert lib.hsa_selftest_wait_timeout(1000, vp(FAKE), n - 1, None) == WORKSPACE
    assert lib.hsa_selftest_wait_timeout(0, vp(FAKE), n, None) == INVALID
    assert lib.hsa_kernel_launches() == before


def test_decode_noalloc_checks_the_size_before_the_memory(lib):
    # an oversized shape is refused for its size even when the memory pointers
    # are pageable host memory (which a fitting shape would have refused)
    np = pytest.importorskip("numpy")
    vp = ctypes.c_void_p
    host = np.zeros(1 << 16, np.uint8)
    hp = (host.ctypes.data + 15) // 16 * 16
    big = hsa.DecodeShape(Bq=1024, Hq=8, Hkv=1, d=128, n_chunks=1 << 20).c()
    args = [vp(FAKE), vp(hp), vp(hp), vp(FAKE), vp(FAKE), vp(FAKE), vp(FAKE), vp(FAKE)]
    assert lib.hsa_decode_noalloc(ctypes.byref(big), *args, None) == WORKSPACE


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    import paper_2504_16795_gb300.binding as b
    monkeypatch.setattr(b, "_lib", None)
    monkeypatch.setattr(b._build, "LIB", str(tmp_path / "absent.so"))
    with pytest.raises(RuntimeError, match="not built"):
        b.load()


def test_memory_append_binding_checks_its_rows(lib):
    torch = pytest.importorskip("torch")
    shape = hsa.DecodeShape(Bq=1, Hq=8, Hkv=2, d=64, n_chunks=0, capacity_chunks=10)
    good = torch.zeros((5, 2, 64), dtype=torch.bfloat16)
    for bad in (torch.zeros((5, 2, 64), dtype=torch.float32), torch.zeros((5, 1, 64), dtype=torch.bfloat16),
                torch.zeros((5, 2, 128), dtype=torch.bfloat16)[..., ::2]):
        with pytest.raises(ValueError):
            hsa.memory_append(shape, 0, bad, good, good, good, good)
        with pytest.raises(ValueError):
            hsa.memory_append(shape, 0, good, bad, good, good, good)
