"""GPU parity of the projection kernel (frt_gemm_bf16) and of the DiT-block attention
slice (frt_block_step) against the fp64 oracle, through the C ABI.

Tolerances. Projection: fp32 accumulation of K bf16 products; whatever the summation
order the error is at most about K * 2^-24 * sum_k |a_ik b_jk|, tested with K * 2^-23;
a bf16 output adds half an ulp of the result (2^-9 relative) before it. Stored q, k, v:
the GPU rounds its fp32 sum to bf16, the oracle its fp64 sum, so an element may differ
by one bf16 ulp where the sum lies near a rounding boundary (rare). Attention output and
block output: the chunk-attention tolerance (max |err| 2e-2, rel-L2 5e-3).
"""

import numpy as np
import pytest
import torch

from oracle.frt_oracle import OracleBlock, bf16_round, linear
from paper_2607_18171_gb300 import synth

from .parity_util import MAX_ABS, MAX_REL_L2, assert_close, compare, sample_rows

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def frt():
    from paper_2607_18171_gb300 import frt as f
    f.lib()
    return f


def _f64(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def _gemm_bound(a, b):
    K = a.shape[1]
    return K * 2.0 ** -23 * (np.abs(a) @ np.abs(b).T)


@pytest.mark.parametrize("M,N,K", [(128, 256, 64), (300, 200, 136), (1000, 384, 512),
                                   (4680, 1536, 1536), (96, 4608, 1536)])
@pytest.mark.parametrize("out", [torch.float32, torch.bfloat16])
def test_gemm_matches_fp64(frt, M, N, K, out):
    g = torch.Generator().manual_seed(M * 7 + N * 3 + K)
    a = torch.randn(M, K, generator=g).to(torch.bfloat16)
    b = (torch.randn(N, K, generator=g) * K ** -0.5).to(torch.bfloat16)
    ldc = N + 8                                    # padding columns must stay untouched
    c = torch.full((M, ldc), 7.0, dtype=out, device="cuda")
    frt.gemm_bf16(a.cuda(), b.cuda(), c)
    torch.cuda.synchronize()
    got = _f64(c)
    af, bf = _f64(a), _f64(b)
    ref = linear(af, bf)
    bound = _gemm_bound(af, bf)
    if out == torch.bfloat16:
        bound = bound + 2.0 ** -8 * np.abs(ref)
    err = np.abs(got[:, :N] - ref)
    assert np.all(err <= bound + 1e-30), f"max excess {float(np.max(err - bound)):.3e}"
    assert np.all(got[:, N:] == 7.0)


@pytest.mark.parametrize("bn", [128, 192, 256])
@pytest.mark.parametrize("M,N,K", [(300, 200, 136), (1000, 384, 512), (96, 4608, 1536),
                                   (4680, 1536, 1536)])
def test_gemm_every_tile_width_matches_fp64(frt, M, N, K, bn):
    """Every output-column tile width, single CTAs (M <= 128) and CTA pairs, 2D and 3D
    operand views (K % 64), ragged M, N and K against the same bound."""
    g = torch.Generator().manual_seed(M * 5 + N + K + bn)
    a = torch.randn(M, K, generator=g).to(torch.bfloat16)
    b = (torch.randn(N, K, generator=g) * K ** -0.5).to(torch.bfloat16)
    c = torch.full((M, N), 7.0, dtype=torch.float32, device="cuda")
    frt.selftest_gemm_force_bn(bn)
    try:
        assert frt.gemm_plan(M, N)[0] == bn
        frt.gemm_bf16(a.cuda(), b.cuda(), c)
        torch.cuda.synchronize()
    finally:
        frt.selftest_gemm_force_bn(0)
    af, bf = _f64(a), _f64(b)
    err = np.abs(_f64(c) - linear(af, bf))
    bound = _gemm_bound(af, bf)
    assert np.all(err <= bound + 1e-30), f"bn {bn}: max excess {float(np.max(err - bound)):.3e}"


def test_gemm_tile_width_does_not_change_results(frt):
    """Each output sums its products in one order (k-block, 16-deep step) whatever the
    tile width: every width gives the same bits."""
    g = torch.Generator().manual_seed(3)
    a = torch.randn(1000, 1536, generator=g).to(torch.bfloat16).cuda()
    b = torch.randn(960, 1536, generator=g).to(torch.bfloat16).cuda()
    outs = []
    try:
        for bn in (128, 192, 256):
            frt.selftest_gemm_force_bn(bn)
            c = torch.empty(1000, 960, device="cuda")
            frt.gemm_bf16(a, b, c)
            outs.append(c)
        torch.cuda.synchronize()
    finally:
        frt.selftest_gemm_force_bn(0)
    for c in outs[1:]:
        assert torch.equal(outs[0], c)


def test_gemm_is_deterministic(frt):
    g = torch.Generator().manual_seed(1)
    a = torch.randn(777, 640, generator=g).to(torch.bfloat16).cuda()
    b = torch.randn(512, 640, generator=g).to(torch.bfloat16).cuda()
    c1 = torch.empty(777, 512, device="cuda")
    c2 = torch.empty(777, 512, device="cuda")
    frt.gemm_bf16(a, b, c1)
    frt.gemm_bf16(a, b, c2)
    torch.cuda.synchronize()
    assert torch.equal(c1, c2)


def test_gemm_rejects_bad_arguments(frt):
    a = torch.zeros(64, 12, dtype=torch.bfloat16, device="cuda")      # K % 8 != 0
    b = torch.zeros(64, 12, dtype=torch.bfloat16, device="cuda")
    c = torch.zeros(64, 64, device="cuda")
    with pytest.raises(frt.FrtError):
        frt.gemm_bf16(a, b, c)


def _block_stream(frt, wl, out_dtype=torch.float32):
    return frt.Stream(wl.heads, wl.head_dim, wl.grid_h, wl.grid_w, wl.frames, wl.window,
                      split=wl.split, out_dtype=out_dtype)


def _ulp_check(got, ref, what, err, rotated=False):
    """GPU bf16 values against the oracle's, element by element. `err` bounds the
    projection's fp32-vs-fp64 accumulation difference of each element (it scales with
    sum |x||w|, not with the result, so it matters where the sum cancels): the two
    roundings to bf16 then differ by at most one ulp at |ref| + err, plus err. Rotated
    values take the ulp and the error at the scale of their (2j, 2j+1) pair (the
    rotation moves a pair's error inside the pair, preserving its norm) and get two
    ulps (the GPU rounds before and after rotating). Almost all must match exactly."""
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    mag = np.abs(ref)
    if rotated:
        pr = ref.reshape(*ref.shape[:-1], -1, 2)
        mag = np.repeat(np.sqrt(np.sum(pr * pr, axis=-1)), 2, axis=-1).reshape(ref.shape)
        pe = err.reshape(*err.shape[:-1], -1, 2)
        err = np.repeat(np.sum(pe, axis=-1), 2, axis=-1).reshape(err.shape)
    ulp = np.ldexp(1.0, np.frexp(np.maximum(mag + err, 1e-30))[1] - 8)
    diff = np.abs(got - ref)
    bound = ((2.0 if rotated else 1.0) * ulp + err) * 1.0000001
    assert np.all(diff <= bound), f"{what}: {int(np.sum(diff > bound))} beyond the bound"
    frac_equal = float(np.mean(diff == 0))
    assert frac_equal >= 0.99, f"{what}: only {frac_equal:.4f} exactly equal"


def _run_block(frt, wl, chunks, keep=(), rows_for=None):
    """Stream `chunks` chunks through frt_block_step and the oracle; compare `keep`."""
    w_qkv, w_o = synth.block_weights(wl)
    d = wl.heads * wl.head_dim
    st = _block_stream(frt, wl)
    orc = OracleBlock(synth.as_f64(w_qkv), synth.as_f64(w_o), wl.heads, wl.head_dim, wl.grid_h,
                      wl.grid_w, wl.frames, wl.window, wl.split)
    wq, wo = w_qkv.cuda(), w_o.cuda()
    q_buf = torch.empty(wl.n_q, d, dtype=torch.bfloat16, device="cuda")
    o_buf = torch.empty_like(q_buf)
    y = torch.empty(wl.n_q, d, dtype=torch.float32, device="cuda")
    wq_abs = np.abs(synth.as_f64(w_qkv))
    for c in range(chunks):
        x = synth.chunk_x(wl, 0, c)
        slot, ev = st.block_step(x.cuda(), wq, wo, q_buf, o_buf, y)
        st.sync()
        rows = None if rows_for is None else rows_for(c)
        ref = orc.step(synth.as_f64(x), rows=rows)
        assert (slot, ev) == (ref["slot"], ref["evicted"])
        if c not in keep:
            continue
        n = wl.n_q
        err = d * 2.0 ** -23 * (np.abs(synth.as_f64(x)) @ wq_abs.T)     # [n, 3d]
        eq, ek, ev_ = (err[:, i * d:(i + 1) * d] for i in range(3))
        _ulp_check(_f64(q_buf), ref["q_rot"].reshape(n, d), f"q chunk {c}", eq, rotated=True)
        kc, vc = st.cache()
        k_slot = kc[slot * n:(slot + 1) * n].reshape(n, d)
        v_slot = vc[slot * n:(slot + 1) * n].reshape(n, d)
        _ulp_check(_f64(k_slot), ref["k_rot"].reshape(n, d), f"k chunk {c}", ek, rotated=True)
        _ulp_check(_f64(v_slot), ref["v"].reshape(n, d), f"v chunk {c}", ev_)
        sel = slice(None) if rows is None else rows
        o_got = _f64(o_buf)[sel].reshape(-1, wl.heads, wl.head_dim)
        assert_close(o_got, ref["o"], f"o chunk {c}")
        y_got = _f64(y)[sel]
        max_abs, rel = compare(y_got, ref["y"])
        assert np.all(np.isfinite(y_got))
        assert rel <= MAX_REL_L2 and max_abs <= MAX_ABS, f"y chunk {c}: {max_abs:.3e} {rel:.3e}"
    return st


def test_block_tiny_matches_oracle(frt):
    wl = synth.WORKLOADS["blocktiny"]
    _run_block(frt, wl, wl.chunks, keep=set(range(wl.chunks)))


def test_block_1p3b_matches_oracle_on_sampled_rows(frt):
    wl = synth.WORKLOADS["block1p3b"]
    rows = sample_rows(wl.n_q, wl.tokens_per_frame, count=192, seed=7)
    _run_block(frt, wl, wl.chunks, keep={0, wl.chunks - 1}, rows_for=lambda c: rows)


def test_block_equals_projection_then_separate_path(frt):
    """The fused QKV epilogue (bf16 rounding, RoPE, writes into the ring slot) gives
    exactly what a plain bf16 projection followed by frt_rope3d_qk and
    frt_kv_append_evict gives."""
    wl = synth.WORKLOADS["block1p3b"]
    d = wl.heads * wl.head_dim
    w_qkv, w_o = (t.cuda() for t in synth.block_weights(wl))
    fused = _block_stream(frt, wl)
    sep = _block_stream(frt, wl)
    q_buf = torch.empty(wl.n_q, d, dtype=torch.bfloat16, device="cuda")
    o_buf = torch.empty_like(q_buf)
    y = torch.empty(wl.n_q, d, dtype=torch.float32, device="cuda")
    qkv = torch.empty(wl.n_q, 3 * d, dtype=torch.bfloat16, device="cuda")
    for c in range(3):
        x = synth.chunk_x(wl, 0, c).cuda()
        slot, _ = fused.block_step(x, w_qkv, w_o, q_buf, o_buf, y)
        frt.gemm_bf16(x, w_qkv, qkv)
        q, k, v = (qkv[:, i * d:(i + 1) * d].contiguous().view(wl.n_q, wl.heads, wl.head_dim)
                   for i in range(3))
        sep.rope3d_qk(q, k)
        sep.kv_append_evict(k, v)
        fused.sync()
        sep.sync()
        assert torch.equal(q_buf.view(wl.n_q, wl.heads, wl.head_dim), q)
        n = wl.n_q
        for a, b in zip(fused.cache(), sep.cache()):
            assert torch.equal(a[slot * n:(slot + 1) * n], b[slot * n:(slot + 1) * n])
        # attention over the same cache with the same q gives the same o
        out = sep.new_out()
        sep.chunk_attention(q, out)
        sep.sync()
        o_sep = out.to(torch.bfloat16).view(n, d)
        assert torch.equal(o_buf, o_sep)


def test_block_rejects_bad_shapes(frt):
    wl = synth.WORKLOADS["blocktiny"]
    d = wl.heads * wl.head_dim
    st = _block_stream(frt, wl)
    w_qkv, w_o = (t.cuda() for t in synth.block_weights(wl))
    q_buf = torch.empty(wl.n_q, d, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(ValueError):
        st.block_step(torch.empty(wl.n_q, d + 8, dtype=torch.bfloat16, device="cuda"), w_qkv,
                      w_o, q_buf, q_buf.clone(), torch.empty(wl.n_q, d, device="cuda"))
