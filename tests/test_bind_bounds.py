"""The binding bounds (tests/bounds.py) against fp32 arithmetic on the CPU: an independent fp32
FFT (numpy's pocketfft in single precision) stays within the spectral method's bound, and an
fp32 direct sum in j order within the direct bound, on random and bipolar blocks.  This checks
the bounds the GPU parity tests use are not violated by ordinary fp32 implementations of the two
methods (they are worst-case bounds: the observed errors sit far below them)."""
import numpy as np
import pytest

from bounds import bind_error_factor


def exact_bind(x, y, unbind):
    X, Y = np.fft.fft(x.astype(np.float64)), np.fft.fft(y.astype(np.float64))
    return np.real(np.fft.ifft(X * (np.conj(Y) if unbind else Y)))


@pytest.mark.parametrize("L", [64, 256, 1024, 8192])
@pytest.mark.parametrize("kind", ["normal", "bipolar"])
def test_fp32_fft_within_spectral_bound(L, kind):
    rng = np.random.default_rng(L + len(kind))
    n = max(2, 16384 // L)
    if kind == "normal":
        x = rng.normal(size=(n, L)).astype(np.float32)
        y = rng.normal(size=(n, L)).astype(np.float32)
    else:
        x = (rng.integers(0, 2, size=(n, L)) * 2 - 1).astype(np.float32)
        y = (rng.integers(0, 2, size=(n, L)) * 2 - 1).astype(np.float32)
    bound = bind_error_factor(L, "spectral") * np.linalg.norm(x.astype(np.float64), axis=1) * \
        np.linalg.norm(y.astype(np.float64), axis=1)
    for unbind in (False, True):
        X, Y = np.fft.rfft(x), np.fft.rfft(y)
        assert X.dtype == np.complex64
        z = np.fft.irfft(X * (np.conj(Y) if unbind else Y), n=L)
        assert z.dtype == np.float32
        err = np.abs(z.astype(np.float64) - exact_bind(x, y, unbind)).max(axis=1)
        assert np.all(err <= bound)
        assert np.all(err <= bound / 8)  # with room to spare: the bound is a worst case


@pytest.mark.parametrize("L", [8, 64, 256])
def test_fp32_direct_sum_within_direct_bound(L):
    rng = np.random.default_rng(L)
    n = 64
    x = rng.normal(size=(n, L)).astype(np.float32)
    y = rng.normal(size=(n, L)).astype(np.float32)
    k = np.arange(L)
    z = np.zeros((n, L), dtype=np.float32)
    for j in range(L):  # one fp32 sum per output in j order
        z = (z + x[:, j:j + 1] * y[:, (k - j) % L]).astype(np.float32)
    err = np.abs(z.astype(np.float64) - exact_bind(x, y, False)).max(axis=1)
    bound = bind_error_factor(L, "direct") * np.linalg.norm(x.astype(np.float64), axis=1) * \
        np.linalg.norm(y.astype(np.float64), axis=1)
    assert np.all(err <= bound)
