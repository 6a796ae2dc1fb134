"""GPU parity of the Haar kernel bank (Sec. 2.3 DWT-Enhanced Architecture) against the
oracle, through the C-ABI: forward level, inverse level, both band counts, fp32 and bf16,
the vector path (W a multiple of 4) and the scalar path, and a VAE-sized feature map."""
import numpy as np
import pytest
import torch

import oracle
from paper_2605_15684_gb300 import api, build, synthetic

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    build.build()
    api.load_library()


def _x(shape, dtype, seed):
    return synthetic.feature_map(*shape, dtype=dtype, seed=seed)


U = 2.0 ** -24  # fp32 unit roundoff


def _mag_dwt(x, nb):
    """Half the sum of |inputs| of each window: bounds every band's fp32 rounding error."""
    N, C, H, W = x.shape
    m = 0.5 * np.abs(x).reshape(N, C, H // 2, 2, W // 2, 2).sum(axis=(3, 5))
    return np.concatenate([m] * nb, axis=1)


def _mag_iwt(y, C, nb):
    N, _, h, w = y.shape
    m = 0.5 * np.abs(y).reshape(N, nb, C, h, w).sum(axis=1)
    return np.repeat(np.repeat(m, 2, axis=2), 2, axis=3)


def _check(got, ref, mag, dtype):
    """fp32: three roundings of a four-term sum (the halving is exact); bf16: both sides read
    the same bf16 inputs, so the only further loss is the bf16 rounding of the result."""
    got = got.float().cpu().double().numpy()
    tol = 4 * U * mag + (2.0 ** -8 * np.abs(ref) if dtype == torch.bfloat16 else 0.0)
    err = np.abs(got - ref)
    assert np.all(err <= tol), f"max excess {float(np.max(err - tol)):.3e}"


# vector path: W a multiple of 8 (bf16) or 4 (fp32); the others take the scalar path
SHAPES = [(1, 1, 2, 2), (2, 3, 16, 16), (1, 5, 34, 18), (1, 4, 10, 4), (2, 16, 258, 260), (1, 7, 66, 130),
          (1, 3, 6, 24), (3, 2, 12, 40), (2, 9, 130, 136)]


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("nb", [4, 3])
@pytest.mark.parametrize("shape", SHAPES)
def test_dwt_matches_oracle(shape, nb, dtype):
    x = _x(shape, dtype, seed=sum(shape) + nb)
    y = api.haar_dwt(x.cuda(), nb=nb)
    torch.cuda.synchronize()
    xd = x.double().numpy()
    _check(y, oracle.haar_dwt(xd, nb), _mag_dwt(xd, nb), dtype)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("nb", [4, 3])
@pytest.mark.parametrize("shape", SHAPES)
def test_iwt_matches_oracle(shape, nb, dtype):
    N, C, H, W = shape
    y = _x((N, nb * C, H // 2, W // 2), dtype, seed=7 * sum(shape) + nb)
    x = api.haar_iwt(y.cuda(), C, nb=nb)
    torch.cuda.synchronize()
    yd = y.double().numpy()
    _check(x, oracle.haar_iwt(yd, C, nb), _mag_iwt(yd, C, nb), dtype)


def test_round_trip_is_identity_fp32():
    x = _x((2, 8, 128, 96), torch.float32, seed=3).cuda()
    back = api.haar_iwt(api.haar_dwt(x), 8)
    torch.cuda.synchronize()
    assert torch.allclose(back, x, rtol=0, atol=32 * U * float(x.abs().max()))


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_vae_sized_feature_map(dtype):
    """A 1024x1024 map of 16 channels: many grid-stride rounds per thread."""
    x = _x((1, 16, 1024, 1024), dtype, seed=11)
    y = api.haar_dwt(x.cuda(), nb=4)
    torch.cuda.synchronize()
    xd = x.double().numpy()
    _check(y, oracle.haar_dwt(xd, 4), _mag_dwt(xd, 4), dtype)
    back = api.haar_iwt(y, 16, nb=4)
    torch.cuda.synchronize()
    yd = y.double().cpu().numpy()
    _check(back, oracle.haar_iwt(yd, 16, 4), _mag_iwt(yd, 16, 4), dtype)


def test_into_caller_buffers_and_stream():
    x = _x((1, 3, 32, 32), torch.float32, seed=5).cuda()
    y = torch.full((1, 9, 16, 16), float("nan"), device="cuda")
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        api.haar_dwt(x, nb=3, y=y, stream=s)
    s.synchronize()
    xd = x.double().cpu().numpy()
    _check(y, oracle.haar_dwt(xd, 3), _mag_dwt(xd, 3), torch.float32)


PYR_SHAPES = [(1, 1, 8, 8), (2, 3, 16, 24), (1, 5, 24, 40), (2, 2, 32, 12), (1, 16, 256, 264), (1, 4, 4, 4)]


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("nb", [4, 3])
@pytest.mark.parametrize("levels", [1, 2, 3])
@pytest.mark.parametrize("shape", PYR_SHAPES)
def test_pyramid_matches_oracle(shape, levels, nb, dtype):
    N, C, H, W = shape
    if H % (1 << levels) or W % (1 << levels):
        pytest.skip("sizes not divisible by 2^levels")
    x = _x(shape, dtype, seed=31 * sum(shape) + levels)
    ys = api.haar_dwt_pyramid(x.cuda(), levels, nb=nb)
    torch.cuda.synchronize()
    refs = oracle.haar_dwt_pyramid(x.double().numpy(), levels, nb)
    # level l's rounding bound: the sum of |x| over its 2^l x 2^l tile, halved l times, with one
    # rounding per level on the way (bf16 rounds the LL it passes down only in the output)
    xa = np.abs(x.double().numpy())
    for l, (got, ref) in enumerate(zip(ys, refs), start=1):
        t = 1 << l
        tile = xa.reshape(N, C, H // t, t, W // t, t).sum(axis=(3, 5)) / 2 ** l
        mag = np.concatenate([tile] * nb, axis=1) * (1 + 2 * l)
        _check(got, ref, mag, dtype)
    # the inverse pyramid on the oracle's bands (rounded to dtype)
    yin = [torch.from_numpy(r).to(dtype) for r in refs]
    back = api.haar_iwt_pyramid([t.cuda() for t in yin], C, nb=nb)
    torch.cuda.synchronize()
    ydn = [t.double().numpy() for t in yin]
    ref_back = oracle.haar_iwt_pyramid(ydn, C, nb)
    mag = sum(np.repeat(np.repeat(0.5 * np.abs(y).reshape(N, nb, C, *y.shape[2:]).sum(axis=1), 1 << l, axis=2),
                        1 << l, axis=3) for l, y in enumerate(ydn, start=1)) * 4
    _check(back, ref_back, mag, dtype)


def test_pyramid_round_trip_fp32_and_ignored_ll():
    x = _x((2, 6, 64, 48), torch.float32, seed=9).cuda()
    ys = api.haar_dwt_pyramid(x, 3)
    ys[0][:, :6] = 1e6  # shallower LL bands are not read by the inverse
    ys[1][:, :6] = -1e6
    back = api.haar_iwt_pyramid(ys, 6)
    torch.cuda.synchronize()
    assert torch.allclose(back, x, rtol=0, atol=64 * U * float(x.abs().max()))
