"""The debug-bounds build (compiled with HSA_DEBUG_BOUNDS) on the GPU.

It runs in a child process that loads _build_debug/libhsa_debug.so:
- On clean inputs, the forward and backward results equal the normal
  library's bit for bit, and hsa_check reports HSA_OK.
- With a planted out-of-range index, the call still completes, and the next
  hsa_check reports HSA_ERR_BOUNDS. The planted indices are:
  a chunk id past the sequence in idx (seen by the forward, the backward and
  the inverse index); an inverted pair of offsets (a list that ends before it
  starts); a slot id past the end in entries.

Every planted value is harmless even to the normal build. Out-of-range chunk
ids count as no selection; an inverted list is empty; with G = 8 the query
rows of any slot id stay inside q, and the partial rows go out by TMA stores,
which drop rows past the tensor. So the test shows that the checks report
these values; it does not rely on them to prevent a fault.
"""
import json
import os
import subprocess
import sys

import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover - collected on CPU only with -m gpu
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2504_16795_gb300 as hsa  # noqa: E402
import synth  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
WORKLOAD = dict(B=1, L=64 * 40 + 9, S=64, Hq=16, Hkv=2, d=128, topk=4)


def run_case(lib_path, case):
    """One case, in whichever library the binding was pointed at; returns (check status, result digest)."""
    import hashlib

    w = synth.Workload("debug-bounds", 91, **WORKLOAD)
    shape = hsa.Shape(B=w.B, L=w.L, Hq=w.Hq, Hkv=w.Hkv, d=w.d, topk=w.topk)
    X = {n: synth.device_tensor(w, n) for n in ("q", "K", "V", "dO")}
    wss = hsa.Workspaces(shape, X["q"].device)
    fwd = hsa.hsa_forward_path(shape, X["q"], X["K"], X["V"], wss)
    idx, offsets, entries = fwd["idx"].clone(), fwd["offsets"].clone(), fwd["entries"].clone()
    n_slots = idx.numel()
    if case == "idx":  # a chunk id past the sequence
        idx.view(-1)[n_slots // 2] = shape.Nc + 5
    elif case == "offsets":  # a list that ends before it starts
        k = offsets.numel() // 2
        offsets[k] = offsets[k + 1] + 3
    elif case == "entries":  # a slot id past the end
        entries[entries.numel() // 3] = n_slots + 7
    torch.cuda.synchronize()
    hsa.check(wss.select)
    hsa.check(wss.forward)
    O, wts = fwd["O"].clone(), fwd["w"].clone()
    hsa.forward(shape, X["q"], X["K"], X["V"], idx, fwd["s_sel"], offsets, entries, O, wts, ws=wss.forward)
    dq, dK, dV = hsa.backward(shape, X["q"], X["K"], X["V"], fwd["kbar32"], idx, wts, O, X["dO"], offsets, entries,
                              ws=wss.backward)
    # the inverse index of the (possibly planted) selection, in its own workspace
    hsa.check(wss.index)
    hsa.build_index(shape, idx, ws=wss.index)
    torch.cuda.synchronize()
    codes = {}
    for name in ("forward", "backward", "index"):
        ws = getattr(wss, name)
        codes[name] = int(hsa.load().hsa_check(ws.data_ptr(), ws.numel(), None))
    h = hashlib.sha256()
    for t in (O, wts, dq, dK, dV):
        h.update(t.contiguous().view(torch.uint8).cpu().numpy().tobytes())
    return codes, h.hexdigest()


CHILD = r"""
import json, os, sys
sys.path.insert(0, {root!r})
sys.path.insert(0, os.path.join({root!r}, "tests"))
import paper_2504_16795_gb300.binding as bnd
from paper_2504_16795_gb300.build import build
bnd._build.LIB = build(debug_bounds=True)
import test_gpu_debug_bounds as t
out = {{c: t.run_case(bnd._build.LIB, c) for c in ("clean", "idx", "offsets", "entries")}}
print("RESULT " + json.dumps(out))
"""


@pytest.fixture(scope="module")
def debug_results():
    r = subprocess.run([sys.executable, "-c", CHILD.format(root=ROOT)], capture_output=True, text=True,
                       timeout=900, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-3000:]
    line = [x for x in r.stdout.splitlines() if x.startswith("RESULT ")][-1]
    return json.loads(line[len("RESULT "):])


def test_debug_build_matches_the_normal_build_on_clean_inputs(debug_results):
    hsa.build()
    codes, digest = run_case(None, "clean")
    assert codes == {"forward": 0, "backward": 0, "index": 0}
    dbg_codes, dbg_digest = debug_results["clean"]
    assert dbg_codes == {"forward": 0, "backward": 0, "index": 0}
    assert dbg_digest == digest


@pytest.mark.parametrize("case", ["idx", "offsets", "entries"])
def test_debug_build_reports_planted_indices(debug_results, case):
    BOUNDS = 6
    codes, _ = debug_results[case]
    # the planted index reaches the forward (its index-free merge reads idx, its chunk
    # kernel reads offsets and entries) and the backward (the same inputs)
    assert codes["forward"] == BOUNDS, codes
    assert codes["backward"] == BOUNDS, codes
    # the index reads idx alone: only a chunk id past the sequence reaches it
    assert codes["index"] == (BOUNDS if case == "idx" else 0), codes
