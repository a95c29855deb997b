"""Pins for the fp64 oracle: each check ties it to something other than itself
(brute force, closed forms, invariants, library routines), and the mutation
tests at the end plant plausible mistakes in copies of the oracle to show
that some pin catches each of them. CPU only."""

import itertools
import math

import numpy as np
import pytest
import torch

import oracle.frt_oracle as O
from paper_2607_18171_gb300 import synth

RNG = np.random.default_rng(12345)


# ---------------------------------------------------------------------------
# reusable checks (each returns the max deviation; a pin passes when it is tiny)
# ---------------------------------------------------------------------------
def full_sequence_bruteforce(qs, ks, vs, window, scale):
    """Pure-Python loops: full-sequence attention with the block-causal mask
    M[i,j] = 1 iff chunk(i) - W < chunk(j) <= chunk(i). qs/ks/vs: lists of
    per-chunk [Nq,H,D] arrays (already rotated). Returns per-chunk outputs."""
    n_chunks = len(qs)
    nq, nh, dim = qs[0].shape
    tok_q = [(c, i) for c in range(n_chunks) for i in range(nq)]
    outs = [np.zeros((nq, nh, dim)) for _ in range(n_chunks)]
    for (ci, i) in tok_q:
        for h in range(nh):
            keys = [(cj, j) for (cj, j) in tok_q if ci - window < cj <= ci]
            sc = []
            for (cj, j) in keys:
                dot = 0.0
                for d in range(dim):
                    dot += qs[ci][i, h, d] * ks[cj][j, h, d]
                sc.append(scale * dot)
            m = max(sc)
            ex = [math.exp(s - m) for s in sc]
            z = sum(ex)
            for d in range(dim):
                acc = 0.0
                for (w, (cj, j)) in zip(ex, keys):
                    acc += w * vs[cj][j, h, d]
                outs[ci][i, h, d] = acc / z
    return outs


def full_sequence_masked(qs, ks, vs, window, scale):
    """One full-sequence pass with a materialised block-causal mask (numpy)."""
    nq = qs[0].shape[0]
    q = np.concatenate(qs)
    k = np.concatenate(ks)
    v = np.concatenate(vs)
    chunk_of = np.repeat(np.arange(len(qs)), nq)
    mask = (chunk_of[None, :] <= chunk_of[:, None]) & (chunk_of[None, :] > chunk_of[:, None] - window)
    out = np.empty_like(q)
    for h in range(q.shape[1]):
        s = scale * np.einsum("id,jd->ij", q[:, h], k[:, h])
        s = np.where(mask, s, -np.inf)
        s = s - s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p /= p.sum(axis=1, keepdims=True)
        out[:, h] = p @ v[:, h]
    return np.split(out, len(qs))


def run_stream(stream_cls, shape, n_chunks, seed, exact=True):
    heads, dim, gh, gw, frames, window = shape
    st = stream_cls(heads, dim, gh, gw, frames, window, synth.default_split(dim), exact=exact)
    qs, ks, vs, outs, idx = [], [], [], [], []
    for c in range(n_chunks):
        q, k, v = (synth.as_f64(t) for t in synth.random_qkv(st.n_q, heads, dim, [seed, c]))
        q_r, k_r = st.rope(q, k)
        slot, ev = st.append(k_r, v)
        outs.append(st.attend(q_r))
        qs.append(q_r), ks.append(k_r), vs.append(v)
        idx.append((slot, ev))
    return qs, ks, vs, outs, idx, st


def max_dev(a_list, b_list):
    return max(float(np.max(np.abs(a - b))) for a, b in zip(a_list, b_list))


# ---------------------------------------------------------------------------
# bf16 rounding
# ---------------------------------------------------------------------------
def test_bf16_round_matches_torch_float32_conversion():
    x = np.concatenate([
        RNG.standard_normal(20000).astype(np.float32),
        (RNG.standard_normal(5000) * 1e30).astype(np.float32),
        (RNG.standard_normal(5000) * 1e-38).astype(np.float32),  # bf16 subnormals
        np.array([0.0, -0.0, 3.3895314e38, -3.3895314e38, 1.0e-45], np.float32),
    ])
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    got = O.bf16_round(x.astype(np.float64))
    assert np.array_equal(got, ref)


def test_bf16_round_ties_to_even():
    # 1 + 2^-8 is halfway between 1 and 1 + 2^-7 -> even (1.0)
    assert O.bf16_round(1.0 + 2.0**-8) == 1.0
    # 1 + 3*2^-8 is halfway between 1 + 2^-7 (odd) and 1 + 2^-6 (even)
    assert O.bf16_round(1.0 + 3 * 2.0**-8) == 1.0 + 2.0**-6
    assert O.bf16_round(-(1.0 + 2.0**-8 + 2.0**-30)) == -(1.0 + 2.0**-7)
    assert np.isinf(O.bf16_round(3.5e38))


# ---------------------------------------------------------------------------
# RoPE
# ---------------------------------------------------------------------------
SPLIT = (16, 24, 24)


def test_rope_identity_at_origin():
    x = RNG.standard_normal((1, 3, 64))
    y = O.rope3d(x, 0, 4, 4, 3, SPLIT)
    assert np.array_equal(x, y)  # token 0 of chunk 0 sits at (0, 0, 0)


def test_rope_preserves_pair_and_vector_norms():
    x = RNG.standard_normal((48, 2, 64))
    y = O.rope3d(x, 5, 4, 4, 3, SPLIT)
    pn = lambda a: a[..., 0::2] ** 2 + a[..., 1::2] ** 2
    assert np.max(np.abs(pn(x) - pn(y))) < 1e-12
    assert np.max(np.abs(np.linalg.norm(x, axis=-1) - np.linalg.norm(y, axis=-1))) < 1e-12


def test_rope_closed_form_frequencies_and_axes():
    """Unit vectors in one pair: position (t,h,w) turns pair j of segment a by
    exactly pos_a * 10000**(-2j/d_a) and leaves the other segments alone."""
    gh, gw, F = 4, 4, 3
    # token index of frame f, row r, col c inside a chunk
    tok = lambda f, r, c: f * gh * gw + r * gw + c
    cases = [
        # (chunk, f, r, c, segment offset, width, pair j, expected position)
        (0, 1, 0, 0, 0, 16, 0, 1.0),      # t = 1, pair 0 -> 1 rad
        (0, 1, 0, 0, 0, 16, 1, 1.0),      # t = 1, pair 1 -> 10000^(-1/8)
        (2, 0, 0, 0, 0, 16, 7, 6.0),      # t = 2*3 + 0 = 6, last t pair
        (0, 0, 2, 0, 16, 24, 0, 2.0),     # h = 2, pair 0 -> 2 rad
        (0, 0, 3, 1, 16, 24, 5, 3.0),     # h = 3
        (0, 0, 1, 3, 40, 24, 0, 3.0),     # w = 3, pair 0 -> 3 rad
        (1, 2, 3, 2, 40, 24, 11, 2.0),    # w = 2, last w pair
    ]
    for chunk, f, r, c, off, width, j, pos in cases:
        x = np.zeros((gh * gw * F, 1, 64))
        i = tok(f, r, c)
        x[i, 0, off + 2 * j] = 1.0
        y = O.rope3d(x, chunk, gh, gw, F, SPLIT)
        phi = pos * 10000.0 ** (-2.0 * j / width)
        expect = np.zeros(64)
        expect[off + 2 * j] = math.cos(phi)
        expect[off + 2 * j + 1] = math.sin(phi)
        assert np.max(np.abs(y[i, 0] - expect)) < 1e-14, (chunk, f, r, c, off, j)
    # 10000^(-1/8) written out: 0.31622776601683794
    x = np.zeros((48, 1, 64)); x[tok(1, 0, 0), 0, 2] = 1.0
    y = O.rope3d(x, 0, gh, gw, F, SPLIT)
    assert abs(y[tok(1, 0, 0), 0, 2] - math.cos(0.31622776601683794)) < 1e-15


def test_rope_complex_multiplication_crosscheck():
    """Independent formulation: each pair as a complex number times e^{i phi},
    with phi built from an explicit per-token loop over (t, h, w)."""
    gh, gw, F, chunk = 3, 5, 2, 4
    x = RNG.standard_normal((gh * gw * F, 2, 64))
    y = O.rope3d(x, chunk, gh, gw, F, SPLIT)
    z = x[..., 0::2] + 1j * x[..., 1::2]   # [tok, H, 32]
    phis = np.zeros((x.shape[0], 32))
    for i in range(x.shape[0]):
        f, rem = divmod(i, gh * gw)
        r, c = divmod(rem, gw)
        pos = (chunk * F + f, r, c)
        col = 0
        for a, width in enumerate(SPLIT):
            for j in range(width // 2):
                phis[i, col] = pos[a] / (10000.0 ** (2 * j / width))
                col += 1
    zr = z * np.exp(1j * phis)[:, None, :]
    assert np.max(np.abs(y[..., 0::2] - zr.real)) < 1e-12
    assert np.max(np.abs(y[..., 1::2] - zr.imag)) < 1e-12


def test_rope_logits_depend_only_on_relative_position():
    gh, gw, F = 4, 4, 3
    q = RNG.standard_normal((48, 2, 64))
    k = RNG.standard_normal((48, 2, 64))
    def logits(cq, ck):
        a = O.rope3d(q, cq, gh, gw, F, SPLIT)
        b = O.rope3d(k, ck, gh, gw, F, SPLIT)
        return np.einsum("ihd,jhd->hij", a, b)
    # chunk shift: (2, 0) vs (5, 3) vs (9, 7)
    l0, l1, l2 = logits(2, 0), logits(5, 3), logits(9, 7)
    assert np.max(np.abs(l0 - l1)) < 1e-10 and np.max(np.abs(l0 - l2)) < 1e-10
    # spatial shift inside a frame: same content vectors at shifted tokens
    x = RNG.standard_normal((1, 1, 64)); w = RNG.standard_normal((1, 1, 64))
    xx = np.repeat(x, 48, 0); ww = np.repeat(w, 48, 0)
    a = O.rope3d(xx, 1, gh, gw, F, SPLIT)[:, 0]
    b = O.rope3d(ww, 1, gh, gw, F, SPLIT)[:, 0]
    tok = lambda f, r, c: f * 16 + r * 4 + c
    base = a[tok(0, 0, 1)] @ b[tok(2, 1, 0)]
    shifted = a[tok(0, 2, 3)] @ b[tok(2, 3, 2)]   # both shifted by (0, +2, +2)
    assert abs(base - shifted) < 1e-10


# ---------------------------------------------------------------------------
# attention + cache
# ---------------------------------------------------------------------------
TINY_SHAPES = [
    # heads, dim, gh, gw, frames, window
    (1, 8, 2, 2, 1, 2),
    (2, 8, 1, 3, 2, 3),
    (1, 12, 2, 1, 3, 1),
    (2, 8, 1, 1, 1, 3),     # one token per chunk (the GPU's one-token edge case)
]


@pytest.mark.parametrize("shape", TINY_SHAPES)
def test_stream_matches_pure_python_bruteforce(shape):
    n_chunks = 4
    # generic split for small head dims: (d/4, 3d/8, 3d/8) rounded to even
    qs, ks, vs, outs, _, st = run_stream(O.OracleStream, shape, n_chunks, 7)
    bf = full_sequence_bruteforce(qs, ks, vs, shape[5], st.scale)
    assert max_dev(outs, bf) < 1e-12


def test_chunked_with_cache_equals_full_sequence_pass():
    shape = (2, 64, 4, 4, 3, 3)  # the tiny workload's shape
    qs, ks, vs, outs, _, st = run_stream(O.OracleStream, shape, 6, 99)
    full = full_sequence_masked(qs, ks, vs, 3, st.scale)
    assert max_dev(outs, full) < 1e-12


def test_softmax_rows_sum_to_one():
    shape = (2, 64, 4, 4, 3, 3)
    qs, ks, vs, outs, _, st = run_stream(O.OracleStream, shape, 4, 3)
    _, p = st.attend(qs[-1], return_probs=True)
    assert np.max(np.abs(p.sum(axis=-1) - 1.0)) < 1e-12
    assert p.min() >= 0.0 and p.max() <= 1.0


def test_window_one_equals_torch_sdpa_float64():
    shape = (2, 16, 2, 3, 2, 1)
    qs, ks, vs, outs, _, st = run_stream(O.OracleStream, shape, 3, 5)
    for q, k, v, o in zip(qs, ks, vs, outs):
        t = lambda a: torch.from_numpy(a).permute(1, 0, 2)[None]  # [1,H,N,D]
        ref = torch.nn.functional.scaled_dot_product_attention(t(q), t(k), t(v))
        ref = ref[0].permute(1, 0, 2).numpy()
        assert np.max(np.abs(ref - o)) < 1e-12


def test_closed_form_equal_keys_give_mean_of_values():
    nq, nkv, nh, d = 5, 11, 2, 8
    q = RNG.standard_normal((nq, nh, d))
    k = np.repeat(RNG.standard_normal((1, nh, d)), nkv, axis=0)
    v = RNG.standard_normal((nkv, nh, d))
    out = O.attention(q, k, v, 0.3)
    assert np.max(np.abs(out - v.mean(axis=0)[None])) < 1e-13


def test_closed_form_one_hot_values_give_softmax_column():
    nq, nkv, nh = 4, 6, 1
    q = RNG.standard_normal((nq, nh, 8))
    k = RNG.standard_normal((nkv, nh, 8))
    v = np.zeros((nkv, nh, nkv)); v[np.arange(nkv), 0, np.arange(nkv)] = 1.0
    out = O.attention(q, k, v, 0.5)
    s = 0.5 * q[:, 0] @ k[:, 0].T
    p = np.exp(s) / np.exp(s).sum(axis=1, keepdims=True)
    assert np.max(np.abs(out[:, 0] - p)) < 1e-14


def test_sampled_rows_equal_full_rows():
    q = RNG.standard_normal((40, 2, 8)); k = RNG.standard_normal((70, 2, 8)); v = RNG.standard_normal((70, 2, 8))
    full = O.attention(q, k, v, 0.35)
    rows = np.array([0, 7, 39, 13])
    assert np.array_equal(O.attention(q, k, v, 0.35, rows=rows), full[rows])


# ---------------------------------------------------------------------------
# indices
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("window", [1, 2, 3, 7])
def test_window_indices_closed_form_and_deque(window):
    st = O.OracleStream(1, 8, 1, 2, 1, window, (2, 2, 4), exact=True)
    z = np.zeros((2, 1, 8))
    for c in range(51):
        slot, ev = st.append(z, z)
        assert slot == c % window
        assert ev == (c - window if c >= window else -1)
        held = [e[0] for e in st.cache]
        assert held == list(range(max(0, c - window + 1), c + 1))
        assert st.cached_kv()[0].shape[0] == min(c + 1, window) * 2


# ---------------------------------------------------------------------------
# mutation tests: plausible mistakes planted in copies of the oracle
# ---------------------------------------------------------------------------
def _rope_copy(x, chunk, gh, gw, F, split, theta=10000.0, sign=1.0, swap_hw=False, exp_factor=2.0):
    """Copy of the oracle's rotation with switchable planted mistakes."""
    x = np.asarray(x, np.float64)
    f, r, col = O.token_positions(chunk, x.shape[0], gh, gw)
    if swap_hw:
        r, col = col, r
    out = x.copy()
    off = 0
    for pos, width in ((chunk * F + f, split[0]), (r, split[1]), (col, split[2])):
        j = np.arange(width // 2)
        ang = np.outer(pos, theta ** (-exp_factor * j / width))[:, None, :]
        x0 = x[:, :, off:off + width:2]
        x1 = x[:, :, off + 1:off + width:2]
        out[:, :, off:off + width:2] = x0 * np.cos(ang) - sign * x1 * np.sin(ang)
        out[:, :, off + 1:off + width:2] = x0 * np.sin(ang) + x1 * np.cos(ang)
        off += width
    return out


def test_rope_copy_without_mistakes_matches_oracle():
    x = RNG.standard_normal((48, 2, 64))
    assert np.max(np.abs(_rope_copy(x, 3, 4, 4, 3, SPLIT) - O.rope3d(x, 3, 4, 4, 3, SPLIT))) < 1e-15


@pytest.mark.parametrize("kw", [dict(swap_hw=True), dict(exp_factor=1.0)])
def test_mutant_rope_is_caught_by_closed_form_pin(kw, monkeypatch):
    monkeypatch.setattr(O, "rope3d", lambda *a: _rope_copy(*a, **kw))
    with pytest.raises(AssertionError):
        test_rope_closed_form_frequencies_and_axes()


def test_mutant_rope_sign_is_caught_by_norm_pin(monkeypatch):
    monkeypatch.setattr(O, "rope3d", lambda *a: _rope_copy(*a, sign=-1.0))
    with pytest.raises(AssertionError):
        test_rope_preserves_pair_and_vector_norms()


class _StreamKeepsOneExtraChunk(O.OracleStream):
    def append(self, k_rot, v):  # mistake: evicts only when len > W + 1
        slot, evicted, _ = O.window_index(self.chunk, self.window)
        self.cache.append((self.chunk, k_rot, v))
        if len(self.cache) > self.window + 1:
            self.cache.popleft()
        self.chunk += 1
        return slot, evicted


class _StreamDropsScale(O.OracleStream):
    def attend(self, q_rot, rows=None, return_probs=False):
        k, v = self.cached_kv()
        return O.attention(q_rot, k, v, 1.0, rows=rows, return_probs=return_probs)


class _StreamAttendsTransposed(O.OracleStream):
    def attend(self, q_rot, rows=None, return_probs=False):
        k, v = self.cached_kv()
        # mistake: values taken from K (a swapped operand)
        return O.attention(q_rot, k, k, self.scale, rows=rows, return_probs=return_probs)


@pytest.mark.parametrize("mutant", [_StreamKeepsOneExtraChunk, _StreamDropsScale, _StreamAttendsTransposed])
def test_mutant_streams_are_caught_by_bruteforce(mutant):
    shape = (1, 8, 2, 2, 1, 2)
    qs, ks, vs, outs, _, st = run_stream(mutant, shape, 4, 7)
    bf = full_sequence_bruteforce(qs, ks, vs, shape[5], 1.0 / math.sqrt(8))
    assert max_dev(outs, bf) > 1e-6


# ---------------------------------------------------------------------------
# the stored-precision branch: rotated q and k rounded to bf16 (exact=False),
# which is what every GPU parity test compares against
# ---------------------------------------------------------------------------
def _bf16_round_bits(x: float) -> float:
    """Round one float64 to the nearest bfloat16 value, ties to even, by integer
    arithmetic on its IEEE-754 bit pattern (independent of the oracle's frexp / rint
    route). Inputs here are normal and far from the overflow edge."""
    import struct
    if x == 0.0:
        return x
    bits = struct.unpack("<Q", struct.pack("<d", x))[0]
    sign = bits >> 63
    exp = (bits >> 52) & 0x7FF
    mant = (bits & ((1 << 52) - 1)) | (1 << 52)        # 53 significant bits
    drop = 53 - 8                                       # keep 8 significant bits
    keep, rest = mant >> drop, mant & ((1 << drop) - 1)
    half = 1 << (drop - 1)
    if rest > half or (rest == half and (keep & 1)):
        keep += 1
    value = math.ldexp(keep, exp - 1075 + drop)
    return -value if sign else value


def _rotate_pure_python(x, chunk, gh, gw, frames, split, theta=10000.0):
    """3D RoPE written token by token and pair by pair with the math module."""
    nq, nh, dim = x.shape
    out = np.array(x, dtype=np.float64)
    tpf = gh * gw
    for i in range(nq):
        f, rem = divmod(i, tpf)
        r, col = divmod(rem, gw)
        pos = (chunk * frames + f, r, col)
        off = 0
        for a in range(3):
            width = split[a]
            for j in range(width // 2):
                ang = pos[a] * math.pow(theta, -2.0 * j / width)
                c, s = math.cos(ang), math.sin(ang)
                for h in range(nh):
                    x0 = float(x[i, h, off + 2 * j])
                    x1 = float(x[i, h, off + 2 * j + 1])
                    out[i, h, off + 2 * j] = x0 * c - x1 * s
                    out[i, h, off + 2 * j + 1] = x0 * s + x1 * c
            off += width
    return out


def _bf16_pure_python(a):
    return np.vectorize(_bf16_round_bits, otypes=[np.float64])(a)


def test_bf16_bit_rounding_helper_matches_torch():
    """The helper above is itself checked against torch's fp32 -> bf16 conversion on
    fp32-representable inputs (where one rounding is all there is), ties included."""
    x = np.concatenate([RNG.standard_normal(4000).astype(np.float32),
                        np.array([1.0 + 2.0**-8, 1.0 + 3 * 2.0**-8, -(1.0 + 2.0**-8)],
                                 np.float32)])
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(_bf16_pure_python(x.astype(np.float64)), ref)


def _stored_precision_reference(shape, n_chunks, seed):
    """Per chunk: independently rotated, independently bf16-rounded q and k, and v."""
    heads, dim, gh, gw, frames, window = shape
    split = synth.default_split(dim)
    qs, ks, vs = [], [], []
    for c in range(n_chunks):
        q, k, v = (synth.as_f64(t) for t in synth.random_qkv(frames * gh * gw, heads, dim, [seed, c]))
        qs.append(_bf16_pure_python(_rotate_pure_python(q, c, gh, gw, frames, split)))
        ks.append(_bf16_pure_python(_rotate_pure_python(k, c, gh, gw, frames, split)))
        vs.append(v)
    return qs, ks, vs


def _run_stored_precision(stream_cls, shape, n_chunks, seed):
    heads, dim, gh, gw, frames, window = shape
    st = stream_cls(heads, dim, gh, gw, frames, window, synth.default_split(dim), exact=False)
    outs = []
    for c in range(n_chunks):
        q, k, v = (synth.as_f64(t) for t in synth.random_qkv(st.n_q, heads, dim, [seed, c]))
        outs.append(st.step(q, k, v)[0])
    return outs, st


@pytest.mark.parametrize("shape", TINY_SHAPES)
def test_stored_precision_stream_matches_bruteforce_on_rounded_rotations(shape):
    """OracleStream(exact=False) rounds the rotated q and k to bf16 before attending
    (they are stored in bf16). Its outputs equal the pure-Python full-sequence brute
    force fed with bf16(rotate(q)), bf16(rotate(k)) built independently."""
    n_chunks = 4
    qs, ks, vs = _stored_precision_reference(shape, n_chunks, 21)
    outs, st = _run_stored_precision(O.OracleStream, shape, n_chunks, 21)
    bf = full_sequence_bruteforce(qs, ks, vs, shape[5], st.scale)
    assert max_dev(outs, bf) < 1e-12
    # and the cache holds exactly the rounded rotated keys, in window order
    k_cached, _ = st.cached_kv()
    assert np.array_equal(k_cached, np.concatenate(ks[max(0, n_chunks - shape[5]):]))


class _StreamLeavesKUnrounded(O.OracleStream):
    def rope(self, q, k):   # mistake: only q is rounded
        args = (self.chunk, self.grid_h, self.grid_w, self.frames_per_chunk, self.split, self.theta)
        return O.bf16_round(O.rope3d(q, *args)), O.rope3d(k, *args)


class _StreamRoundsBeforeRotating(O.OracleStream):
    def rope(self, q, k):   # mistake: rounds the inputs, then rotates
        args = (self.chunk, self.grid_h, self.grid_w, self.frames_per_chunk, self.split, self.theta)
        return O.rope3d(O.bf16_round(q), *args), O.rope3d(O.bf16_round(k), *args)


@pytest.mark.parametrize("mutant", [_StreamLeavesKUnrounded, _StreamRoundsBeforeRotating])
def test_mutant_rounding_orders_are_caught(mutant):
    shape = (2, 8, 1, 3, 2, 3)
    qs, ks, vs = _stored_precision_reference(shape, 4, 21)
    outs, st = _run_stored_precision(mutant, shape, 4, 21)
    bf = full_sequence_bruteforce(qs, ks, vs, shape[5], st.scale)
    assert max_dev(outs, bf) > 1e-6
