"""Pins of the oracle's streaming causal 3D convolution against things other than
itself: pure-Python brute force on tiny inputs, streamed-with-cache equal to one pass
over the whole sequence, reductions to numpy.convolve (temporal-only kernel) and to the
identity (centre tap), and exact linearity. Planted mistakes in copies of the oracle
must fail a pin."""

import numpy as np
import pytest

import oracle.frt_oracle as O


def _brute(x_ext, w, b, kt, kh, kw):
    n_ext, H, W, cin = x_ext.shape
    F = n_ext - (kt - 1)
    cout = w.shape[1]
    y = np.zeros((F, H, W, cout))
    for t in range(F):
        for h in range(H):
            for x_ in range(W):
                for o in range(cout):
                    acc = float(b[o])
                    for dt in range(kt):
                        for dh in range(kh):
                            for dw in range(kw):
                                hh, ww = h + dh - kh // 2, x_ + dw - kw // 2
                                if 0 <= hh < H and 0 <= ww < W:
                                    tap = (dt * kh + dh) * kw + dw
                                    for c in range(cin):
                                        acc += w[tap, o, c] * x_ext[t + dt, hh, ww, c]
                    y[t, h, x_, o] = acc
    return y


@pytest.mark.parametrize("kt,kh,kw", [(3, 3, 3), (2, 3, 1), (1, 1, 1), (3, 1, 3)])
def test_conv_matches_brute_force(kt, kh, kw):
    rng = np.random.default_rng([kt, kh, kw])
    F, H, W, cin, cout = 2, 4, 5, 3, 2
    x_ext = rng.standard_normal((kt - 1 + F, H, W, cin))
    w = rng.standard_normal((kt * kh * kw, cout, cin))
    b = rng.standard_normal(cout)
    got = O.causal_conv3d(x_ext, w, b, kt, kh, kw)
    assert np.max(np.abs(got - _brute(x_ext, w, b, kt, kh, kw))) <= 1e-12


def _run_stream(cls, chunks, F, seed=0, kt=3, kh=3, kw=3):
    rng = np.random.default_rng(seed)
    H, W, cin, cout = 4, 5, 3, 2
    w = rng.standard_normal((kt * kh * kw, cout, cin))
    b = rng.standard_normal(cout)
    xs = [rng.standard_normal((F, H, W, cin)) for _ in range(chunks)]
    st = cls(cin, cout, kt, kh, kw, H, W)
    ys = [st.step(x, w, b) for x in xs]
    return xs, w, b, ys


@pytest.mark.parametrize("F", [1, 2, 3])
def test_streamed_equals_one_pass_over_the_sequence(F):
    kt = 3
    xs, w, b, ys = _run_stream(O.OracleConvStream, 4, F, seed=F)
    seq = np.concatenate(xs, axis=0)
    ext = np.concatenate([np.zeros((kt - 1,) + seq.shape[1:]), seq], axis=0)
    whole = O.causal_conv3d(ext, w, b, kt, 3, 3)
    assert np.max(np.abs(np.concatenate(ys, axis=0) - whole)) <= 1e-12


def test_temporal_only_kernel_is_numpy_convolve():
    """kh = kw = 1, one channel in and out: each pixel's series is a causal 1D convolution."""
    rng = np.random.default_rng(7)
    kt, T, H, W = 3, 6, 2, 3
    x = rng.standard_normal((T, H, W, 1))
    k = rng.standard_normal(kt)
    w = k.reshape(kt, 1, 1)            # tap dt weights frame t + dt - (kt - 1) by k[dt]
    ext = np.concatenate([np.zeros((kt - 1, H, W, 1)), x], axis=0)
    y = O.causal_conv3d(ext, w, np.zeros(1), kt, 1, 1)
    for h in range(H):
        for c in range(W):
            series = x[:, h, c, 0]
            # y[t] = sum_dt k[dt] x[t + dt - (kt - 1)] = (series * k reversed)[t]
            ref = np.convolve(series, k[::-1])[:T]
            assert np.max(np.abs(y[:, h, c, 0] - ref)) <= 1e-12


def test_centre_tap_identity_returns_the_input():
    rng = np.random.default_rng(8)
    kt, kh, kw, C = 3, 3, 3, 4
    x = rng.standard_normal((2, 5, 6, C))
    w = np.zeros((kt * kh * kw, C, C))
    w[((kt - 1) * kh + 1) * kw + 1] = np.eye(C)   # newest frame, centre pixel
    ext = np.concatenate([np.zeros((kt - 1, 5, 6, C)), x], axis=0)
    assert np.array_equal(O.causal_conv3d(ext, w, np.zeros(C), kt, kh, kw), x)


def test_linearity_in_weights_and_input():
    rng = np.random.default_rng(9)
    ext = rng.standard_normal((4, 3, 4, 2))
    w1, w2 = rng.standard_normal((2, 27, 3, 2))
    b = np.zeros(3)
    a = O.causal_conv3d(ext, w1 + w2, b, 3, 3, 3)
    s = O.causal_conv3d(ext, w1, b, 3, 3, 3) + O.causal_conv3d(ext, w2, b, 3, 3, 3)
    assert np.max(np.abs(a - s)) <= 1e-12
    assert np.array_equal(O.causal_conv3d(2.0 * ext, w1, b, 3, 3, 3),
                          2.0 * O.causal_conv3d(ext, w1, b, 3, 3, 3))


# ---- planted mistakes --------------------------------------------------------------------

class _StreamKeepsNewestFirst(O.OracleConvStream):
    def step(self, x, w, bias):
        y = super().step(x, w, bias)
        self.cache = self.cache[::-1].copy()      # frame order reversed in the cache
        return y


class _StreamForgetsCache(O.OracleConvStream):
    def step(self, x, w, bias):
        y = super().step(x, w, bias)
        self.cache = np.zeros_like(self.cache)
        return y


def _flipped_conv(x_ext, w, bias, kt, kh, kw):
    return O.causal_conv3d(x_ext, w[::-1].copy(), bias, kt, kh, kw)   # taps reversed


@pytest.mark.parametrize("mutant", [_StreamKeepsNewestFirst, _StreamForgetsCache])
def test_mutant_streams_fail_the_one_pass_pin(mutant):
    xs, w, b, ys = _run_stream(mutant, 4, 1, seed=3)
    seq = np.concatenate(xs, axis=0)
    ext = np.concatenate([np.zeros((2,) + seq.shape[1:]), seq], axis=0)
    whole = O.causal_conv3d(ext, w, b, 3, 3, 3)
    assert np.max(np.abs(np.concatenate(ys, axis=0) - whole)) > 1e-6


def test_mutant_tap_order_fails_the_brute_force_pin():
    rng = np.random.default_rng(4)
    x_ext = rng.standard_normal((4, 3, 4, 2))
    w = rng.standard_normal((27, 2, 2))
    b = np.zeros(2)
    assert np.max(np.abs(_flipped_conv(x_ext, w, b, 3, 3, 3) - _brute(x_ext, w, b, 3, 3, 3))) > 1e-6
