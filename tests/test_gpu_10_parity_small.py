"""GPU vs fp64 oracle on sizes the oracle finishes in seconds: every output element,
several tiles, ragged tails; fused vs separate paths; determinism; indices."""

import numpy as np
import pytest
import torch

from paper_2607_18171_gb300 import synth
from tests import parity_util as U

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def frt():
    from paper_2607_18171_gb300 import frt as m
    m.lib()
    return m


SMALL = {
    # ragged: Nq = 3*130 = 390 (second 256-row item has one partial tile), Nkv up to 1170
    "ragged_d128": synth.Workload("ragged_d128", 90, 1, 3, 128, 10, 13, 3, 3, 5, (32, 48, 48)),
    # one frame per chunk, Nq = 7*19 = 133 (tile 2 holds 5 rows), window 4, per-head scales
    "ragged_scaled": synth.Workload("ragged_scaled", 91, 1, 2, 128, 7, 19, 1, 4, 6, (32, 48, 48),
                                    head_scale=True),
    # head_dim 64 beyond one KV tile: Nq = 2*80 = 160, window 2 -> Nkv 320
    "d64_multi_tile": synth.Workload("d64_multi_tile", 92, 1, 3, 64, 8, 10, 2, 2, 4, (16, 24, 24)),
    # window 1: plain bidirectional attention per chunk
    "window1": synth.Workload("window1", 93, 1, 2, 128, 5, 9, 2, 1, 3, (32, 48, 48)),
    # the widest token row the library accepts: heads * head_dim = 12800 (25.6 KB rows)
    "max_row": synth.Workload("max_row", 94, 1, 100, 128, 4, 5, 2, 2, 3, (32, 48, 48)),
    # the smallest chunk: one token (1 x 1 grid, one frame); Nkv 1..3, far below one tile
    "one_token": synth.Workload("one_token", 95, 1, 2, 64, 1, 1, 1, 3, 5, (16, 24, 24)),
    # mixed work split on 152 SMs: 80 heads x 2 query groups (Nq 280) = 160 groups, 152
    # run whole and the last 8 are cut into KV parts (the dit1p3b / 720p plan, small)
    "mixed_split_d128": synth.Workload("mixed_split_d128", 98, 1, 80, 128, 7, 20, 2, 2, 3,
                                       (32, 48, 48)),
    # the same at head_dim 64: 160 heads x one 256-row group, window 3
    "mixed_split_d64": synth.Workload("mixed_split_d64", 99, 1, 160, 64, 8, 16, 2, 3, 4,
                                      (16, 24, 24)),
}


@pytest.mark.parametrize("name", ["mixed_split_d128", "mixed_split_d64"])
def test_mixed_split_cases_plan_whole_and_cut_groups(frt, name):
    """The two cases above keep their purpose: on this GPU, at a full window, some query
    groups run whole and the rest are cut into KV parts merged on the device."""
    wl = SMALL[name]
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    n_full, n_split = frt.attention_plan([wl.n_q], [wl.window * wl.n_q], wl.heads, sms)
    assert n_full > 0 and n_split > 1, (n_full, n_split)


@pytest.mark.parametrize("name", ["tiny"] + list(SMALL))
@pytest.mark.parametrize("fused", [True, False])
def test_stream_matches_oracle_every_element(frt, name, fused):
    wl = synth.WORKLOADS.get(name) or SMALL[name]
    st = U.make_stream(wl, frt)
    run = U.run_fused if fused else U.run_separate
    got = run(st, wl, 0, wl.chunks, keep=range(wl.chunks))
    ref = U.oracle_full_stream(wl, 0, wl.chunks)
    for c in range(wl.chunks):
        out, slot, ev = got[c]
        r_out, r_slot, r_ev = ref[c]
        assert (slot, ev) == (r_slot, r_ev)
        U.assert_close(out, r_out, f"{name} chunk {c}")
    st.close()


@pytest.mark.parametrize("name", ["tiny", "ragged_d128"])
def test_fused_and_separate_paths_are_bit_identical(frt, name):
    wl = synth.WORKLOADS.get(name) or SMALL[name]
    a = U.make_stream(wl, frt)
    b = U.make_stream(wl, frt)
    ra = U.run_fused(a, wl, 0, wl.chunks, keep=range(wl.chunks))
    rb = U.run_separate(b, wl, 0, wl.chunks, keep=range(wl.chunks))
    for c in range(wl.chunks):
        assert np.array_equal(ra[c][0], rb[c][0]), f"chunk {c}"
    ka, va = a.cache()
    kb, vb = b.cache()
    assert torch.equal(ka.view(torch.int16), kb.view(torch.int16))
    assert torch.equal(va.view(torch.int16), vb.view(torch.int16))
    a.close(); b.close()


def test_run_to_run_determinism(frt):
    wl = SMALL["ragged_d128"]
    outs = []
    for _ in range(2):
        st = U.make_stream(wl, frt)
        outs.append(U.run_fused(st, wl, 0, wl.chunks, keep=range(wl.chunks)))
        st.close()
    for c in range(wl.chunks):
        assert np.array_equal(outs[0][c][0], outs[1][c][0])


def test_reset_restarts_the_stream_bit_identically(frt):
    """After reset (cache, counter, split-KV merge counters, status cleared) a stream
    reproduces a fresh stream's outputs bit for bit."""
    wl = SMALL["ragged_d128"]
    fresh = U.make_stream(wl, frt)
    ref = U.run_fused(fresh, wl, 0, wl.chunks, keep=range(wl.chunks))
    fresh.close()
    st = U.make_stream(wl, frt)
    U.run_fused(st, wl, 1, 2)            # other inputs first
    st.reset()
    got = U.run_fused(st, wl, 0, wl.chunks, keep=range(wl.chunks))
    for c in range(wl.chunks):
        assert got[c][1:] == ref[c][1:]
        assert np.array_equal(got[c][0], ref[c][0]), f"chunk {c}"
    st.close()


def test_failed_configure_leaves_the_stream_unconfigured(frt):
    import ctypes
    L = frt.lib()
    # accepted shape (Nq = 2^20, W * Nq = 2^24, heads * head_dim = 12800) whose cache,
    # 2 x 430 GB, no GPU holds: the allocation fails cleanly with FRT_ERR_OOM
    h = L.frt_stream_create(100, 128, 1 << 16, 16, 16)
    assert h
    cfg = frt.Config()
    assert L.frt_config_default(h, ctypes.byref(cfg)) == 0
    assert L.frt_stream_configure(h, ctypes.byref(cfg)) == 3          # FRT_ERR_OOM
    buf = ctypes.create_string_buffer(64)
    p = ctypes.cast(buf, ctypes.c_void_p)
    assert L.frt_rope3d_qk(h, p, p) == 2                              # FRT_ERR_STATE
    assert L.frt_stream_reset(h) == 2
    L.frt_stream_destroy(h)
    torch.cuda.synchronize()                                         # the context is fine


def test_bf16_output(frt):
    wl = SMALL["ragged_d128"]
    st = U.make_stream(wl, frt, out_dtype=torch.bfloat16)
    got = U.run_fused(st, wl, 0, wl.chunks, keep=range(wl.chunks))
    ref = U.oracle_full_stream(wl, 0, wl.chunks)
    for c in range(wl.chunks):
        U.assert_close(got[c][0], ref[c][0], f"bf16 chunk {c}")
    st.close()


def test_rope_within_one_bf16_ulp_of_oracle(frt):
    from oracle.frt_oracle import bf16_round, rope3d
    wl = SMALL["ragged_d128"]
    st = U.make_stream(wl, frt)
    for c in range(3):
        q, k, v = synth.chunk_qkv(wl, 0, c)
        qd, kd = q.cuda(), k.cuda()
        st.rope3d_qk(qd, kd)
        st.kv_append_evict(kd, v.cuda())
        args = (c, wl.grid_h, wl.grid_w, wl.frames, wl.split)
        for got, src in ((qd, q), (kd, k)):
            x = synth.as_f64(src)
            ref = bf16_round(rope3d(x, *args))
            g = got.float().cpu().numpy().astype(np.float64)
            ulp = np.ldexp(1.0, np.frexp(np.maximum(np.abs(ref), 1e-30))[1] - 8)
            # fp32 rotation with fp32 cos/sin: absolute error <= ~3 * 2^-24 * |pair|,
            # which exceeds one bf16 ulp of the result only under cancellation
            pair = np.sqrt(x[..., 0::2] ** 2 + x[..., 1::2] ** 2).repeat(2, axis=-1)
            bound = ulp + 2.0**-21 * pair
            assert np.all(np.abs(g - ref) <= bound), float(np.max(np.abs(g - ref) / bound))
            assert np.mean(g == ref) > 0.99
    st.close()


def test_append_writes_slot_bytes_and_evicts_whole_chunks(frt):
    wl = SMALL["ragged_d128"]
    st = U.make_stream(wl, frt)
    kept = {}
    for c in range(7):
        q, k, v = U.gpu_inputs(wl, 0, c)
        st.rope3d_qk(q, k)
        slot, ev = st.kv_append_evict(k, v)
        assert slot == c % wl.window and ev == (c - wl.window if c >= wl.window else -1)
        kept[c] = (k.clone(), v.clone())
    st.sync()
    kc, vc = st.cache()
    nq = wl.n_q
    for c in range(7 - wl.window, 7):
        s = c % wl.window
        assert torch.equal(kc[s * nq:(s + 1) * nq].view(torch.int16), kept[c][0].view(torch.int16))
        assert torch.equal(vc[s * nq:(s + 1) * nq].view(torch.int16), kept[c][1].view(torch.int16))
    st.close()


def test_batched_ragged_streams_match_single_launches_and_oracle(frt):
    base = SMALL["ragged_d128"]
    fills = [3, 1, 2, 3]
    streams, outs_b, outs_s, qs = [], [], [], []
    for s, fill in enumerate(fills):
        st = U.make_stream(base, frt)
        for c in range(fill - 1):
            q, k, v = U.gpu_inputs(base, s, c)
            st.chunk_step(q, k, v, st.new_out())
        q, k, v = U.gpu_inputs(base, s, fill - 1)
        st.rope3d_qk(q, k)
        st.kv_append_evict(k, v)
        streams.append(st); qs.append(q)
        outs_b.append(st.new_out())
    frt.chunk_attention_batched(streams, qs, outs_b)
    for st, q in zip(streams, qs):
        o = st.new_out()
        st.chunk_attention(q, o)
        outs_s.append(o)
    torch.cuda.synchronize()
    for s, fill in enumerate(fills):
        # the two launches may pick different split-KV factors (the batched one sees
        # more query groups); each split rounds P to bf16 against its own running max,
        # so the two agree to the bf16 rounding of P, not bit for bit
        max_abs, rel = U.compare(outs_b[s].cpu().numpy(), outs_s[s].cpu().numpy())
        assert max_abs <= 5e-3 and rel <= 2e-3, (s, max_abs, rel)
        ref = U.oracle_full_stream(base, s, fill)[fill - 1][0]
        U.assert_close(outs_b[s].cpu().numpy(), ref, f"stream {s}")
    for st in streams:
        st.close()


def test_batched_at_the_stream_limit(frt):
    """32 streams, the most one batched launch takes, with fills 1..W, against the oracle."""
    base = synth.WORKLOADS["tiny"]
    fills = [1 + s % base.window for s in range(32)]
    streams, qs, outs = [], [], []
    for s, fill in enumerate(fills):
        st = U.make_stream(base, frt)
        for c in range(fill - 1):
            q, k, v = U.gpu_inputs(base, s, c)
            st.chunk_step(q, k, v, st.new_out())
        q, k, v = U.gpu_inputs(base, s, fill - 1)
        st.rope3d_qk(q, k)
        st.kv_append_evict(k, v)
        streams.append(st)
        qs.append(q)
        outs.append(st.new_out())
    frt.chunk_attention_batched(streams, qs, outs)
    torch.cuda.synchronize()
    for s, fill in enumerate(fills):
        ref = U.oracle_full_stream(base, s, fill)[fill - 1][0]
        U.assert_close(outs[s].cpu().numpy(), ref, f"stream {s}")
    for st in streams:
        st.close()


def test_host_buffer_step_pipelined_matches_device_path_and_oracle(frt):
    """frt_chunk_step_host keeps several chunks in flight (copy-in, compute and
    copy-out overlap across calls); after one sync every chunk's output must equal
    the device-buffer path bit for bit and match the oracle."""
    wl = SMALL["ragged_d128"]
    a = U.make_stream(wl, frt)
    b = U.make_stream(wl, frt)
    host_outs = []
    for c in range(wl.chunks):
        q, k, v = (t.pin_memory() for t in synth.chunk_qkv(wl, 0, c))
        o = torch.empty(a.shape(), dtype=torch.float32).pin_memory()
        a.chunk_step_host(q, k, v, o)
        host_outs.append((o, q, k, v))   # keep host buffers alive until the sync
    a.sync()
    dev = U.run_fused(b, wl, 0, wl.chunks, keep=range(wl.chunks))
    ref = U.oracle_full_stream(wl, 0, wl.chunks)
    for c in range(wl.chunks):
        got = host_outs[c][0].numpy()
        assert np.array_equal(got, dev[c][0]), c
        U.assert_close(got, ref[c][0], f"host path chunk {c}")
    a.close(); b.close()


@pytest.mark.parametrize("scale_last", [20.0, 0.05])
def test_scores_growing_or_shrinking_across_tiles(frt, scale_last):
    """Keys of the newest chunk scaled up (scores far above every earlier tile: the
    kernel's stale exponent reference must be replaced and O rescaled) or down (later
    tiles far below the reference): the result still matches the oracle."""
    from oracle.frt_oracle import OracleStream
    wl = SMALL["ragged_d128"]
    st = U.make_stream(wl, frt)
    orc = OracleStream(wl.heads, wl.head_dim, wl.grid_h, wl.grid_w, wl.frames, wl.window,
                       wl.split)
    for c in range(wl.window):
        q, k, v = synth.chunk_qkv(wl, 0, c)
        if c == wl.window - 1:
            k = (k.float() * scale_last).to(torch.bfloat16)
        ref = orc.step(synth.as_f64(q), synth.as_f64(k), synth.as_f64(v))[0]
        qd, kd, vd = q.cuda(), k.cuda(), v.cuda()
        out = st.new_out()
        st.chunk_step(qd, kd, vd, out)
        st.sync()
        got = out.cpu().numpy()
        assert np.all(np.isfinite(got))
        U.assert_close(got, ref, f"chunk {c} scale {scale_last}")
    st.close()
