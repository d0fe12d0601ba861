"""sbd_linear (y = x W^T on the LM-head kernel, used to time full forwards
around the block step) against the oracle's fp64 product: every element
within bf16 output rounding plus the fp32 accumulation bound."""
import numpy as np
import pytest

import gen
import oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sbd():
    import paper_2509_04185_gb300 as m
    return m


def _bf16(rng, shape, scale):
    return gen.f32_to_bf16_bits((rng.standard_normal(shape) * scale).astype(np.float32))


@pytest.mark.parametrize("T,K,N", [(1, 4096, 6144), (5, 64, 1), (16, 256, 129), (17, 256, 1000),
                                   (64, 4096, 128), (100, 512, 777), (128, 1024, 2048),
                                   (200, 256, 300), (256, 4096, 4096), (300, 128, 129),
                                   (512, 256, 1000),
                                   # few rows, narrow layers: K split over CTAs
                                   (16, 4096, 4096), (2, 14336, 512), (64, 1024, 300),
                                   # above 160 rows: CTA pairs (one or two row
                                   # groups; narrow layers with K ranges)
                                   (161, 64, 1), (193, 64, 1), (257, 128, 513), (384, 1024, 257),
                                   (512, 4096, 6144), (512, 14336, 4096), (256, 14336, 512),
                                   (320, 4096, 4096)])
def test_matches_fp64_product(sbd, T, K, N):
    import torch
    rng = np.random.default_rng(T * 7 + N)
    xb, wb = _bf16(rng, (T, K), 1.0), _bf16(rng, (N, K), 0.02)
    x = torch.from_numpy(xb.view(np.int16)).view(torch.bfloat16).cuda()
    w = torch.from_numpy(wb.view(np.int16)).view(torch.bfloat16).cuda()
    y = sbd.sbd_linear(x, w).float().cpu().numpy()
    xf, wf = gen.bf16_bits_to_f32(xb), gen.bf16_bits_to_f32(wb)
    ref = oracle.linear(xf, wf)
    bound = np.abs(xf).astype(np.float64) @ np.abs(wf).astype(np.float64).T
    tol = 2.0 ** -8 * np.abs(ref) + K * 2.0 ** -23 * bound + 1e-6
    assert y.shape == (T, N)
    assert np.all(np.abs(y - ref) <= tol), float(np.max(np.abs(y - ref) - tol))
    assert sbd.sbd_device_error() == 0


def test_out_of_range_rows_are_not_written(sbd):
    import torch
    rng = np.random.default_rng(1)
    x = torch.from_numpy(_bf16(rng, (3, 128), 1.0).view(np.int16)).view(torch.bfloat16).cuda()
    w = torch.from_numpy(_bf16(rng, (200, 128), 0.1).view(np.int16)).view(torch.bfloat16).cuda()
    big = torch.full((5, 200), 7.0, dtype=torch.bfloat16, device="cuda")
    sbd.sbd_linear(x, w, out=big[:3])
    assert torch.all(big[3:] == 7.0)


@pytest.mark.parametrize("case", range(16))
def test_random_shapes(sbd, case):
    """Seeded random shapes on both sides of the CTA-pair threshold (160
    rows): out_features that leave partial tiles, in_features of any number
    of 64-column boxes (K split where the model picks one)."""
    import torch
    rng = np.random.default_rng(500 + case)
    T = int(rng.integers(1, 513))
    K = 64 * int(rng.integers(1, 65))
    N = int(rng.integers(1, 3000))
    xb, wb = _bf16(rng, (T, K), 1.0), _bf16(rng, (N, K), 0.02)
    x = torch.from_numpy(xb.view(np.int16)).view(torch.bfloat16).cuda()
    w = torch.from_numpy(wb.view(np.int16)).view(torch.bfloat16).cuda()
    y = sbd.sbd_linear(x, w).float().cpu().numpy()
    xf, wf = gen.bf16_bits_to_f32(xb), gen.bf16_bits_to_f32(wb)
    ref = oracle.linear(xf, wf)
    bound = np.abs(xf).astype(np.float64) @ np.abs(wf).astype(np.float64).T
    tol = 2.0 ** -8 * np.abs(ref) + K * 2.0 ** -23 * bound + 1e-6
    assert np.all(np.abs(y - ref) <= tol), (T, K, N, float(np.max(np.abs(y - ref) - tol)))
    assert sbd.sbd_device_error() == 0
