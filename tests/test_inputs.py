"""The synthetic input recipes (stand-ins for the paper's gradients, Sec. 5.1): sizes, scales and
determinism as stated, so that every test and bench line draws the same inputs."""
import numpy as np

from paper_2409_17836_gb300 import inputs as I


def test_tiny_gradient_layers_and_seed():
    g = I.tiny_gradient(0)
    assert g.dtype == np.float32 and g.size == 4096
    for l in range(4):
        s = 10.0 ** (-3.0 + 2.0 * l / 3.0)  # 1e-3, 4.64e-3, 2.15e-2, 1e-1
        part = g[1024 * l: 1024 * (l + 1)].astype(np.float64)
        # the sample std of 1024 normals is within 10% of sigma far beyond 5 standard errors
        assert abs(part.std() / s - 1.0) < 0.1, l
        assert abs(part.mean()) < 0.2 * s, l
    assert np.array_equal(g, I.tiny_gradient(0)) and not np.array_equal(g, I.tiny_gradient(1))


def test_convnet_gradient_size_and_determinism():
    g = I.convnet_gradient(0)
    # conv 3*64*9+64, 64*128*9+128, 128*192*9+192, fc 192*10+10
    assert g.size == 1792 + 73856 + 221376 + 1930 == 298954
    assert g.dtype == np.float32 and np.all(np.isfinite(g)) and np.count_nonzero(g) > 0.9 * g.size
    assert np.array_equal(g, I.convnet_gradient(0))
    assert not np.array_equal(g, I.convnet_gradient(1))


def test_laplace_mixture_scales():
    n, t = 200 * 4000, 200
    g = I.laplace_gradient(n=n, n_tensors=t, seed=5)
    assert g.dtype == np.float32 and g.size == n
    b = np.abs(g.astype(np.float64)).reshape(t, -1).mean(axis=1)  # E|x| = b for Laplace(0, b)
    assert b.min() > 0.9e-5 and b.max() < 1.1e-2
    # log10 b is uniform on [-5, -2]: its sample mean is near -3.5
    assert abs(np.log10(b).mean() + 3.5) < 0.25
    last = I.laplace_gradient(n=1000, n_tensors=3, seed=5)
    assert last.size == 1000  # the last tensor takes the remainder (333, 333, 334)
