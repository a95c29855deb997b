"""frt_chunk_attention_noalloc: chunk attention for callers that cannot allocate
device memory (memory planners/arenas that own every device byte, loops where an
allocation is not allowed). It allocates nothing: its split-KV scratch is a static
device array inside the library. Checked here, through the C ABI, against the
allocating entry point frt_chunk_attention on two calls in a row."""

import ctypes

import pytest
import torch

from paper_2607_18171_gb300 import synth
from tests import parity_util as U

pytestmark = pytest.mark.gpu

P, I, D = ctypes.c_void_p, ctypes.c_int, ctypes.c_double


@pytest.fixture(scope="module")
def frt():
    from paper_2607_18171_gb300 import frt as m
    L = m.lib()
    L.frt_chunk_attention_noalloc.restype = I
    L.frt_chunk_attention_noalloc.argtypes = [P, P, P, P, I, I, I, I, D, I, P, P]
    return m


def _call(frt, q, k, v, out, n_q, n_kv, heads, dim, status):
    return frt.lib().frt_chunk_attention_noalloc(
        q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(), n_q, n_kv, heads, dim,
        0.0, 0, status.data_ptr(), torch.cuda.current_stream().cuda_stream)


def test_noalloc_matches_allocating_entry_point_on_two_calls(frt):
    # 4 heads x 128, Nq = 2 * 8 * 32 = 512 (8 query groups), window 8 -> Nkv 4096:
    # the launch splits the KV range, so the static scratch is exercised
    wl = synth.Workload("noalloc", 95, 1, 4, 128, 8, 32, 2, 8, 9, (32, 48, 48))
    st = U.make_stream(wl, frt)
    status = torch.zeros(4, dtype=torch.int32, device="cuda")
    checked = 0
    for c in range(wl.chunks):
        q, k, v = U.gpu_inputs(wl, 0, c)
        st.rope3d_qk(q, k)
        st.kv_append_evict(k, v)
        ref = st.new_out()
        st.chunk_attention(q, ref)
        if c >= wl.chunks - 2:          # two calls in a row, different chunks
            kc, vc = st.cache()
            n_kv = min(c + 1, wl.window) * wl.n_q
            out = torch.full_like(ref, float("nan"))
            rc = _call(frt, q, kc, vc, out, wl.n_q, n_kv, wl.heads, wl.head_dim, status)
            assert rc == 0, frt.lib().frt_last_error().decode()
            torch.cuda.synchronize()
            assert torch.isfinite(out).all()
            max_abs, rel = U.compare(out.cpu().numpy(), ref.cpu().numpy())
            assert max_abs <= 5e-3 and rel <= 2e-3, (c, max_abs, rel)
            checked += 1
    assert checked == 2
    assert int(status.abs().sum()) == 0
    st.close()


def test_noalloc_rejects_sizes_beyond_the_static_maximum(frt):
    t = torch.zeros(16, dtype=torch.bfloat16, device="cuda")
    status = torch.zeros(4, dtype=torch.int32, device="cuda")
    # 1024 heads x ceil(1280 / 256) = 5120 query groups > 4096: rejected before any
    # memory is touched
    rc = _call(frt, t, t, t, t, 1280, 4096, 1024, 128, status)
    assert rc == 5
    assert "4096" in frt.lib().frt_last_error().decode()
