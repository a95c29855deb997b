"""The stream's persistent state (the cross-batch KV-cache edge): snapshot and restore
replay bit-identically, also into another handle (moving the state between resources),
and the guard words around the cache stay intact and are checked on the host."""

import pytest
import torch

from paper_2607_18171_gb300 import synth
from tests import parity_util as U

pytestmark = pytest.mark.gpu

WL = {
    # ragged tails, three chunks past the window
    "ragged": synth.Workload("state_ragged", 80, 1, 3, 128, 10, 13, 3, 3, 6, (32, 48, 48)),
    # 1.3B-like heads and head_dim over a smaller grid: the attention splits its tail
    "split": synth.Workload("state_split", 81, 1, 12, 128, 8, 32, 3, 4, 7, (32, 48, 48)),
    "d64": synth.Workload("state_d64", 82, 1, 2, 64, 4, 4, 3, 3, 6, (16, 24, 24)),
}


@pytest.fixture(scope="module")
def frt():
    from paper_2607_18171_gb300 import frt as m
    m.lib()
    return m


def _steps(st, wl, chunks):
    outs = []
    for c in chunks:
        q, k, v = U.gpu_inputs(wl, 0, c)
        out = st.new_out()
        st.chunk_step(q, k, v, out)
        outs.append(out)
    st.sync()
    return [o.cpu() for o in outs]


@pytest.mark.parametrize("name", list(WL))
def test_restore_replays_bit_identically_in_the_same_and_another_handle(frt, name):
    wl = WL[name]
    cut = wl.window                      # the window is full, chunk 0 already evicted next
    a = U.make_stream(wl, frt)
    _steps(a, wl, range(cut))
    k, v, counter = a.save()
    a.sync()
    assert counter == cut
    first = _steps(a, wl, range(cut, wl.chunks))
    # the same handle, restored
    a.restore(k, v, counter)
    assert a.counter == cut
    again = _steps(a, wl, range(cut, wl.chunks))
    # another handle of the same shape, fresh, restored from the snapshot
    b = U.make_stream(wl, frt)
    b.restore(k, v, counter)
    moved = _steps(b, wl, range(cut, wl.chunks))
    for x, y, z in zip(first, again, moved):
        assert torch.equal(x, y) and torch.equal(x, z)
    # and the replay still matches the oracle
    ref = U.oracle_full_stream(wl, 0, wl.chunks)
    for i, c in enumerate(range(cut, wl.chunks)):
        U.assert_close(first[i].float().numpy(), ref[c][0], f"{name} chunk {c}")
    a.check_guards()
    b.check_guards()
    a.close()
    b.close()


def test_save_refused_between_rope_and_append(frt):
    wl = WL["d64"]
    st = U.make_stream(wl, frt)
    q, k, v = U.gpu_inputs(wl, 0, 0)
    st.rope3d_qk(q, k)
    with pytest.raises(frt.FrtError) as e:
        st.save()
    assert e.value.status == 2
    st.close()


@pytest.mark.parametrize("which", [0, 1, 2, 3])
def test_guard_words_intact_after_streaming_and_a_poke_is_reported(frt, which):
    wl = WL["ragged"]
    st = U.make_stream(wl, frt)
    _steps(st, wl, range(wl.chunks))
    st.check_guards()                                   # every ring write stayed inside
    assert frt.lib().frt_selftest_poke_guard(st.handle, which) == 0
    with pytest.raises(frt.FrtError) as e:
        st.check_guards()
    assert e.value.status == 7
    assert ("before" if which < 2 else "after") in str(e.value)
    assert ("V" if which & 1 else "K") in str(e.value)
    frt.lib().frt_stream_destroy(st.handle)
    st._h = None


def test_release_build_has_no_past_ring_hook(frt):
    if frt.lib().frt_debug_build():
        pytest.skip("debug build")
    assert frt.lib().frt_selftest_append_past_ring() == 5
