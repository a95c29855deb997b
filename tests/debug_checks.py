"""Checks that only run against the FRT_DEBUG build of the library (FRT_LIBRARY=debug),
driven by tests/test_gpu_60_debug_build.py in a child process: the kernels' bounds
checks refuse an access outside the ring and report it, with no trap."""

import pytest
import torch

from paper_2607_18171_gb300 import synth
from tests import parity_util as U

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def frt():
    from paper_2607_18171_gb300 import frt as m
    assert m.lib().frt_debug_build() == 1, "FRT_LIBRARY=debug must load the debug build"
    return m


def test_append_past_the_ring_is_refused_and_reported(frt):
    wl = synth.Workload("debug_ring", 70, 1, 2, 64, 4, 4, 3, 3, 4, (16, 24, 24))
    st = U.make_stream(wl, frt)
    q, k, v = U.gpu_inputs(wl, 0, 0)
    st.chunk_step(q, k, v, st.new_out())
    st.sync()
    assert frt.lib().frt_selftest_append_past_ring() == 0
    q, k, v = U.gpu_inputs(wl, 0, 1)
    st.chunk_step(q, k, v, st.new_out())
    with pytest.raises(frt.FrtError) as e:
        st.sync()
    assert e.value.status == 7 and "bounds" in str(e.value)
    st.check_guards()                 # the refused stores left the guard words intact
    # reset is the way back: the stream reproduces a fresh stream's outputs
    st.reset()
    out = st.new_out()
    st.chunk_step(*U.gpu_inputs(wl, 0, 0), out)
    st.sync()
    ref = U.oracle_full_stream(wl, 0, 1)
    U.assert_close(out.cpu().numpy(), ref[0][0], "after reset")
    st.close()


def test_debug_build_streams_split_and_batched_launches_without_reports(frt):
    # the item checks of the attention kernel on a tail-split launch and a batched one
    wl = synth.Workload("debug_split", 71, 1, 12, 128, 8, 32, 3, 4, 5, (32, 48, 48))
    st = U.make_stream(wl, frt)
    got = U.run_fused(st, wl, 0, wl.chunks, keep=[wl.chunks - 1])
    ref = U.oracle_rows(wl, 0, wl.chunks - 1, list(range(0, wl.n_q, 7)))
    U.assert_close(got[wl.chunks - 1][0][::7], ref, "debug split")
    st.close()
