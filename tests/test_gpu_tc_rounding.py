"""The rounding bound behind the selection certificate, measured on the device.

The tensor-core selection brackets every exact fp32 score by the bf16 score
plus or minus eps_i = 2^-7 (9/8) |q̂| |K̄_i|. Part of that budget is the
rounding of the tensor core's own fp32 accumulation, taken as at most 2^-12
of sum_e |a_e b_e| (plus an absolute floor of 1e-25 for products flushed to
zero). Here the selection's score pass runs on bf16 tiles built to stress
accumulation (random, a wide exponent range, heavy cancellation, one large
product among small ones, values near the bottom of the normal range) and
every result is compared with the exact sum of the exact products.
"""
import math

import numpy as np
import pytest

import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # pragma: no cover - collected on CPU only with -m gpu
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import paper_2504_16795_gb300 as hsa  # noqa: E402

BOUND_REL = 2.0 ** -12
FLOOR_ABS = 1e-25


@pytest.fixture(scope="module", autouse=True)
def built():
    hsa.build()
    hsa.load()


def bf16_bits(x):
    return synth.f32_to_bf16(np.asarray(x, np.float32))


def tiles(kind, d, rng):
    if kind == "normal":
        a, b = rng.standard_normal((128, d)), rng.standard_normal((64, d))
    elif kind == "wide exponents":
        a = rng.standard_normal((128, d)) * 2.0 ** rng.integers(-20, 21, (128, d))
        b = rng.standard_normal((64, d)) * 2.0 ** rng.integers(-20, 21, (64, d))
    elif kind == "cancellation":
        # pairs of products that cancel up to a small remainder
        a = rng.standard_normal((128, d))
        a[:, 1::2] = a[:, 0::2]
        b = rng.standard_normal((64, d))
        b[:, 1::2] = -b[:, 0::2] * (1 + 2.0 ** -7 * rng.integers(-3, 4, (64, d // 2)))
    elif kind == "one large product":
        a = rng.standard_normal((128, d)) * 2.0 ** -10
        b = rng.standard_normal((64, d))
        a[:, rng.integers(0, d, 128)] = 0.0
        a[np.arange(128), rng.integers(0, d, 128)] = 2.0 ** 12
    elif kind == "near the bottom of the range":
        a = rng.standard_normal((128, d)) * 2.0 ** -60
        b = rng.standard_normal((64, d)) * 2.0 ** -62
    else:
        raise ValueError(kind)
    return bf16_bits(a), bf16_bits(b)


KINDS = ["normal", "wide exponents", "cancellation", "one large product", "near the bottom of the range"]


@pytest.mark.parametrize("d", [64, 128])
def test_tensor_core_accumulation_is_within_the_certificate_budget(d):
    rng = np.random.default_rng(d)
    worst = 0.0
    for kind in KINDS:
        for _ in range(2):
            abits, bbits = tiles(kind, d, rng)
            A = torch.from_numpy(abits.view(np.int16)).view(torch.bfloat16).cuda()
            B = torch.from_numpy(bbits.view(np.int16)).view(torch.bfloat16).cuda()
            C = hsa.selftest_score_tile(A, B).cpu().numpy().astype(np.float64)
            a, b = synth.bf16_to_f64(abits), synth.bf16_to_f64(bbits)
            prod = a[:, None, :] * b[None, :, :]  # exact: 8-bit by 8-bit significands
            abs_sum = np.abs(prod).sum(-1)
            exact = np.array([[math.fsum(prod[r, c]) for c in range(64)] for r in range(128)])
            err = np.abs(C - exact)
            assert (err <= BOUND_REL * abs_sum + FLOOR_ABS).all(), (kind, float((err / np.maximum(abs_sum, 1e-300)).max()))
            nz = abs_sum > 1e-20
            if nz.any():
                worst = max(worst, float((err[nz] / abs_sum[nz]).max()))
    # measured worst case, relative to sum |a_e b_e| (reported with -s)
    print(f"d={d}: worst |tensor-core sum - exact| / sum|a_e b_e| = {worst:.3e} (2^{math.log2(max(worst, 1e-300)):.1f})")
    assert worst < BOUND_REL
