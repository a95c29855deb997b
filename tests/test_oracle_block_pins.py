"""Pins of the oracle's DiT-block slice (``linear``, ``OracleBlock``) against things
other than itself: a pure-Python brute-force dot product, permutation weights that turn
every projection into an exact column gather (so the block must reduce to the already
pinned chunk step on permuted inputs), and exact scaling. Mutation tests plant likely
mistakes in copies of the oracle and check that a pin fails for each."""

import numpy as np
import pytest

import oracle.frt_oracle as O

H, D, GH, GW, F, W = 2, 64, 4, 4, 3, 3
SPLIT = (16, 24, 24)
DM = H * D
NQ = F * GH * GW


def _bf16_values(rng, shape, scale=1.0):
    return O.bf16_round(rng.standard_normal(shape) * scale)


def _perm_matrix(perm):
    """Row j has its 1 at column perm[j]: (x @ P^T)[:, j] = x[:, perm[j]]."""
    p = np.zeros((len(perm), len(perm)))
    p[np.arange(len(perm)), perm] = 1.0
    return p


def _perms(rng, n):
    # permutations that are not involutions, so P and P^T act differently
    out = []
    while len(out) < n:
        p = rng.permutation(DM)
        if not np.array_equal(p[p], np.arange(DM)):
            out.append(p)
    return out


def test_linear_matches_pure_python_dot_products():
    rng = np.random.default_rng(5)
    x = rng.standard_normal((3, 5))
    w = rng.standard_normal((4, 5))
    y = O.linear(x, w)
    assert y.shape == (3, 4)
    for i in range(3):
        for j in range(4):
            acc = 0.0
            for t in range(5):
                acc += float(x[i, t]) * float(w[j, t])
            assert abs(y[i, j] - acc) <= 1e-12


def _run_permutation_pin(block_cls, chunks=4, seed=11):
    """Feed a block permutation weights; compare with the chunk step on gathered inputs."""
    rng = np.random.default_rng(seed)
    p_q, p_k, p_v, p_o = _perms(rng, 4)
    w_qkv = np.concatenate([_perm_matrix(p_q), _perm_matrix(p_k), _perm_matrix(p_v)])
    w_o = _perm_matrix(p_o)
    blk = block_cls(w_qkv, w_o, H, D, GH, GW, F, W, SPLIT)
    ref = O.OracleStream(H, D, GH, GW, F, W, SPLIT)
    for c in range(chunks):
        x = _bf16_values(rng, (NQ, DM))
        got = blk.step(x)
        o_ref, slot, ev = ref.step(x[:, p_q].reshape(NQ, H, D), x[:, p_k].reshape(NQ, H, D),
                                   x[:, p_v].reshape(NQ, H, D))
        if not (np.array_equal(got["o"], o_ref) and (got["slot"], got["evicted"]) == (slot, ev)):
            return False
        y_ref = O.bf16_round(o_ref).reshape(NQ, DM)[:, p_o]
        if not np.array_equal(got["y"], y_ref):
            return False
    return True


def test_block_with_permutation_weights_reduces_to_the_chunk_step():
    assert _run_permutation_pin(O.OracleBlock)


def test_block_output_scales_exactly_with_w_o():
    rng = np.random.default_rng(3)
    w_qkv = _bf16_values(rng, (3 * DM, DM), DM ** -0.5)
    w_o = _bf16_values(rng, (DM, DM), DM ** -0.5)
    a = O.OracleBlock(w_qkv, w_o, H, D, GH, GW, F, W, SPLIT)
    b = O.OracleBlock(w_qkv, 2.0 * w_o, H, D, GH, GW, F, W, SPLIT)
    for c in range(2):
        x = _bf16_values(rng, (NQ, DM))
        ya, yb = a.step(x)["y"], b.step(x)["y"]
        assert np.array_equal(2.0 * ya, yb)


def test_block_sampled_rows_equal_full_rows():
    rng = np.random.default_rng(4)
    w_qkv = _bf16_values(rng, (3 * DM, DM), DM ** -0.5)
    w_o = _bf16_values(rng, (DM, DM), DM ** -0.5)
    a = O.OracleBlock(w_qkv, w_o, H, D, GH, GW, F, W, SPLIT)
    b = O.OracleBlock(w_qkv, w_o, H, D, GH, GW, F, W, SPLIT)
    rows = np.array([0, 5, 17, NQ - 1])
    for c in range(3):
        x = _bf16_values(rng, (NQ, DM))
        full, part = a.step(x), b.step(x, rows=rows)
        assert np.array_equal(full["y"][rows], part["y"])


# ---- planted mistakes --------------------------------------------------------------------

class _BlockNoTranspose(O.OracleBlock):
    """Applies the weights as x @ w instead of x @ w^T."""

    def project_qkv(self, x):
        qkv = O.bf16_round(np.asarray(x) @ np.concatenate(
            [self.w_qkv[i * self.d:(i + 1) * self.d] for i in range(3)], axis=1))
        n = qkv.shape[0]
        s = self.stream
        return tuple(qkv[:, i * self.d:(i + 1) * self.d].reshape(n, s.heads, s.head_dim)
                     for i in range(3))


class _BlockSwapsKV(O.OracleBlock):
    def project_qkv(self, x):
        q, k, v = super().project_qkv(x)
        return q, v, k


class _BlockSkipsOutputRounding(O.OracleBlock):
    def step(self, x, rows=None):
        r = super().step(x, rows)
        r["y"] = O.linear(r["o"].reshape(r["o"].shape[0], self.d), self.w_o)
        return r


@pytest.mark.parametrize("mutant", [_BlockNoTranspose, _BlockSwapsKV, _BlockSkipsOutputRounding])
def test_mutant_blocks_are_caught_by_the_permutation_pin(mutant):
    assert not _run_permutation_pin(mutant)
