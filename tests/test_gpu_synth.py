"""The device generator writes bit-for-bit the tensors the host generator draws."""
import numpy as np
import pytest

import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu
if not torch.cuda.is_available():  # pragma: no cover
    pytest.skip("needs a CUDA GPU", allow_module_level=True)


def bits(t):
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


@pytest.mark.parametrize("w", [
    synth.WORKLOADS[1],
    synth.WORKLOADS[2].with_(B=2, L=1024 + 7),
    synth.WORKLOADS[4].with_(L=1 << 14),
    synth.WORKLOADS[5].with_(L=1 << 14, Bq=64, needle_chunks=64),
], ids=["iid", "chunk-offsets", "prefill-needles", "decode-needles"])
def test_device_generator_matches_host(w):
    for name in ("q", "K", "V") + (("dO",) if not w.decode else ()):
        dev = bits(synth.device_tensor(w, name))
        host = synth.host_tensor(w, name, (0, 0, 0, 0), w.dims(name))
        if w.decode:
            host = host[0]
        assert np.array_equal(dev, host), name
