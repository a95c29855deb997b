"""GPU vs fp64 oracle at the full workload sizes, in the launch configuration the
benchmark times (fused frt_chunk_step; batched launch for the multi-stream workload),
on sampled query rows (all heads) that include tile and frame edges and the ragged
tail; plus whole-output properties that hold at any size."""

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


# 720p: chunk 5 is the first full window, chunk 6 the first that evicts (ring slot 0 is
# rewritten while slots 1-5 keep their chunks)
@pytest.mark.parametrize("name,check", [("dit1p3b", [6]), ("dit14b", [0, 6, 19]),
                                        ("stream720p", [5, 6])])
def test_full_size_sampled_rows(frt, name, check):
    wl = synth.WORKLOADS[name]
    n_chunks = max(check) + 1
    st = U.make_stream(wl, frt)
    got = U.run_fused(st, wl, 0, n_chunks, keep=set(check))
    for c in check:
        out, slot, ev = got[c]
        assert (slot, ev) == (c % wl.window, c - wl.window if c >= wl.window else -1)
        assert np.all(np.isfinite(out))
        rows = U.sample_rows(wl.n_q, wl.tokens_per_frame, seed=c)
        ref = U.oracle_rows(wl, 0, c, rows)
        U.assert_close(out[rows], ref, f"{name} chunk {c}")
    st.close()


def test_multi_stream_batched_sampled_rows(frt):
    wl = synth.WORKLOADS["multi8"]
    fills = synth.stream_fills(wl)
    streams, qs, outs = [], [], []
    for s, fill in enumerate(fills):
        st = U.make_stream(wl, frt)
        for c in range(fill - 1):
            q, k, v = U.gpu_inputs(wl, s, c)
            st.chunk_step(q, k, v, st.new_out())
        q, k, v = U.gpu_inputs(wl, s, fill - 1)
        st.rope3d_qk(q, k)
        st.kv_append_evict(k, v)
        streams.append(st); qs.append(q); outs.append(st.new_out())
    frt.chunk_attention_batched(streams, qs, outs)
    torch.cuda.synchronize()
    for s, fill in enumerate(fills):
        rows = U.sample_rows(wl.n_q, wl.tokens_per_frame, count=96, seed=s)
        ref = U.oracle_rows(wl, s, fill - 1, rows)
        out = outs[s].cpu().numpy()
        assert np.all(np.isfinite(out))
        U.assert_close(out[rows], ref, f"multi8 stream {s} fill {fill}")
    for st in streams:
        st.close()


def test_full_size_whole_output_properties(frt):
    """Any size: a chunk whose V is constant per head gives that constant everywhere,
    because the softmax weights sum to 1 -- up to the bf16 rounding of P in the PV
    product (each weight within a relative 2^-9, so the sum within 2^-8)."""
    wl = synth.WORKLOADS["dit1p3b"]
    st = U.make_stream(wl, frt)
    const = torch.linspace(-2, 2, wl.heads)
    for c in range(wl.window):
        q, k, _ = U.gpu_inputs(wl, 0, c)
        v = const.view(1, -1, 1).expand(wl.n_q, wl.heads, wl.head_dim).to(torch.bfloat16)
        out = st.new_out()
        st.chunk_step(q, k, v.contiguous().cuda(), out)
    st.sync()
    ref = const.to(torch.bfloat16).float().view(1, -1, 1)
    assert ((out.cpu() - ref).abs() <= 2.0**-8 * ref.abs() + 1e-6).all()
    st.close()
