"""frt_chunk_attention_noalloc: chunk attention for callers that cannot allocate
device memory (memory planners/arenas that own every device byte, loops where an
allocation is not allowed). It allocates nothing: its split-KV scratch is a static
device array inside the library.

Checked here through the C ABI on two calls in a row per case: element by element
against the fp64 oracle at the contract tolerance (the same rotated q and window),
and against the allocating entry point frt_chunk_attention. The cases make the launch
split the KV range (so the static partials and merge counters are used), one of them
with the partial rows at the array's limit, and one with head_dim 64. Free device
memory must not change across the calls."""

import ctypes

import pytest
import torch

from paper_2607_18171_gb300 import synth
from tests import parity_util as U

pytestmark = pytest.mark.gpu

P, I, D = ctypes.c_void_p, ctypes.c_int, ctypes.c_double

# the static array's partial-row capacity: 8 MiB of fp32 rows and 16384 (max, sum)
# pairs, i.e. groups * split * 256 <= min(8 MiB / (4 * head_dim), 16384)
PART_BYTES = 8 << 20
ML_ROWS = 16384
MAX_SPLIT = 4


def expected_split(groups: int, kv_tiles: int, head_dim: int, sms: int) -> int:
    """The split rule of the entry point written out: the smallest makespan
    ceil(groups * s / SMs) / s * (1 + 0.02 (s - 1)), at least two KV tiles per split,
    and partial rows within the static capacity."""
    cap_rows = min(PART_BYTES // (4 * head_dim), ML_ROWS)
    best, best_t = 1, float(-(-groups // sms))
    for s in range(2, MAX_SPLIT + 1):
        if kv_tiles < 2 * s or groups * s * 256 > cap_rows:
            break
        t = (-(-groups * s // sms)) / s * (1.0 + 0.02 * (s - 1))
        if t < best_t - 1e-9:
            best, best_t = s, t
    return best


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


CASES = [
    # name, seed index, heads, head_dim, grid_w, frames, window, RoPE split
    # 4 heads x 128, Nq 2 * 8 * 32 = 512 (8 query groups), window 8 -> Nkv 4096
    ("d128", 95, 4, 128, 32, 2, 8, (32, 48, 48)),
    # the same at head_dim 64
    ("d64", 96, 4, 64, 32, 2, 8, (16, 24, 24)),
    # 8 heads: 16 groups x 4 splits x 256 = 16384 partial rows, the array's limit
    ("cap", 97, 8, 128, 32, 2, 8, (32, 48, 48)),
]


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_noalloc_matches_oracle_and_allocating_entry_point_on_two_calls(frt, case):
    name, idx, heads, dim, gw, frames, window, split = case
    wl = synth.Workload("noalloc_" + name, idx, 1, heads, dim, 8, gw, frames, window,
                        window + 1, split)
    groups = heads * -(-wl.n_q // 256)
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    split_used = expected_split(groups, -(-(wl.window * wl.n_q) // 128), dim, sms)
    assert split_used > 1, "the case must exercise the static split-KV scratch"
    if name == "cap":
        assert groups * split_used * 256 == ML_ROWS

    st = U.make_stream(wl, frt)
    status = torch.zeros(4, dtype=torch.int32, device="cuda")
    warmed = False
    checked = 0
    for c in range(wl.chunks):
        q, k, v = U.gpu_inputs(wl, 0, c)
        st.rope3d_qk(q, k)
        st.kv_append_evict(k, v)
        ref = st.new_out()
        st.chunk_attention(q, ref)
        if c < wl.chunks - 2:           # two calls in a row: the last two chunks
            continue
        kc, vc = st.cache()
        n_kv = min(c + 1, wl.window) * wl.n_q
        out = torch.empty_like(ref)
        if not warmed:
            # the first call on a device looks up the static array's address
            assert _call(frt, q, kc, vc, out, wl.n_q, n_kv, heads, dim, status) == 0, \
                frt.lib().frt_last_error().decode()
            warmed = True
        out.fill_(float("nan"))
        torch.cuda.synchronize()
        free_before = torch.cuda.mem_get_info()[0]
        rc = _call(frt, q, kc, vc, out, wl.n_q, n_kv, heads, dim, status)
        assert rc == 0, frt.lib().frt_last_error().decode()
        torch.cuda.synchronize()
        assert torch.cuda.mem_get_info()[0] == free_before, "the entry point allocated"
        assert torch.isfinite(out).all()
        got = out.cpu().numpy()
        U.assert_close(got, U.oracle_rows(wl, 0, c, list(range(wl.n_q))),
                       f"{name} chunk {c} vs oracle")
        max_abs, rel = U.compare(got, ref.cpu().numpy())
        assert max_abs <= 5e-3 and rel <= 2e-3, (name, c, max_abs, rel)
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
