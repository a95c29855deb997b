"""C ABI checks that need no GPU: the library builds and loads, exports every symbol
the headers declare, host-side window arithmetic is exact, and argument/state
validation rejects bad calls before any device work."""

import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def frt():
    from paper_2607_18171_gb300 import _build, frt as m
    _build.build()
    m.lib()
    return m


def declared_symbols():
    names = set()
    for h in ("frt.h", "frt_selftest.h"):
        src = open(os.path.join(ROOT, "include", h)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names.update(re.findall(r"\b(frt_[a-z0-9_]+)\s*\(", src))
    return names


def test_library_exports_every_declared_symbol(frt):
    L = frt.lib()
    names = declared_symbols()
    assert {"frt_stream_create", "frt_rope3d_qk", "frt_kv_append_evict",
            "frt_chunk_attention"} <= names
    for n in names:
        assert hasattr(L, n), n


@pytest.mark.parametrize("window", [1, 2, 3, 7])
def test_window_index_bit_exact(frt, window):
    for c in list(range(0, 51)) + [2**31 + 5, 2**40 + 3]:
        slot, ev, valid = frt.window_index(c, window)
        assert slot == c % window
        assert ev == (c - window if c >= window else -1)
        assert valid == min(c + 1, window)


def test_window_index_rejects_bad_args(frt):
    with pytest.raises(frt.FrtError) as e:
        frt.window_index(-1, 3)
    assert e.value.status == 1
    with pytest.raises(frt.FrtError):
        frt.window_index(0, 0)


def test_status_strings(frt):
    L = frt.lib()
    for code, name in frt.STATUS_NAMES.items():
        assert L.frt_status_string(code).decode() == name


def test_create_validates_shapes(frt):
    L = frt.lib()
    assert not L.frt_stream_create(2, 96, 16, 3, 3)
    assert "head_dim" in L.frt_last_error().decode()
    assert not L.frt_stream_create(0, 64, 16, 3, 3)
    assert not L.frt_stream_create(2, 64, 16, 3, 0)
    assert not L.frt_stream_create(2, 64, 1 << 20, 3, 3)
    h = L.frt_stream_create(2, 64, 16, 3, 3)
    assert h
    L.frt_stream_destroy(h)
    # the limits themselves: heads * head_dim <= 12800, Nq <= 2^20, W * Nq <= 2^24
    for args, ok in (((100, 128, 16, 3, 3), True), ((101, 128, 16, 3, 3), False),
                     ((200, 64, 16, 3, 3), True), ((201, 64, 16, 3, 3), False),
                     ((1, 64, 1, 1, 1), True),
                     ((1, 64, 1 << 20, 1, 16), True), ((1, 64, 1 << 20, 1, 17), False),
                     ((1, 64, (1 << 20) + 1, 1, 1), False)):
        h = L.frt_stream_create(*args)
        assert bool(h) == ok, args
        if h:
            L.frt_stream_destroy(h)


def test_configure_rejects_bad_config_before_device_work(frt):
    L = frt.lib()
    h = L.frt_stream_create(2, 64, 16, 3, 3)
    cfg = frt.Config()
    assert L.frt_config_default(h, ctypes.byref(cfg)) == 0
    assert (cfg.rope_dt, cfg.rope_dh, cfg.rope_dw) == (16, 24, 24)
    assert abs(cfg.sm_scale - 0.125) < 1e-15 and cfg.theta == 10000.0
    bad = frt.Config.from_buffer_copy(cfg)
    bad.grid_h, bad.grid_w = 3, 5          # 15 != 16 tokens per frame
    assert L.frt_stream_configure(h, ctypes.byref(bad)) == 1
    bad = frt.Config.from_buffer_copy(cfg)
    bad.grid_h, bad.grid_w = 4, 4
    bad.rope_dt, bad.rope_dh, bad.rope_dw = 15, 25, 24  # odd
    assert L.frt_stream_configure(h, ctypes.byref(bad)) == 1
    bad.rope_dt, bad.rope_dh, bad.rope_dw = 16, 24, 26  # sum != 64
    assert L.frt_stream_configure(h, ctypes.byref(bad)) == 1
    L.frt_stream_destroy(h)


def test_calls_before_configure_are_state_errors(frt):
    L = frt.lib()
    h = L.frt_stream_create(2, 64, 16, 3, 3)
    buf = ctypes.create_string_buffer(64)
    p = ctypes.cast(buf, ctypes.c_void_p)
    assert L.frt_rope3d_qk(h, p, p) == 2
    assert L.frt_kv_append_evict(h, p, p, None, None) == 2
    assert L.frt_chunk_attention(p, None, None, p, h) == 2
    assert L.frt_chunk_step(h, p, p, p, p, None, None) == 2
    assert L.frt_stream_reset(h) == 2
    assert L.frt_stream_chunk_counter(h) == 0
    assert L.frt_rope3d_qk(None, p, p) == 1
    L.frt_stream_destroy(h)
    L.frt_stream_destroy(None)


def test_missing_library_fails_loudly(monkeypatch):
    """No CPU fallback: without libfrt.so the binding raises instead of computing."""
    from paper_2607_18171_gb300 import frt as m
    monkeypatch.setattr(m, "_lib", None)
    monkeypatch.setattr(m, "LIB_PATH", os.path.join(ROOT, "no-such-dir", "libfrt.so"))
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        m.lib()


def test_product_path_does_not_import_the_oracle():
    pkg = os.path.join(ROOT, "paper_2607_18171_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith(".py"):
                src = open(os.path.join(dirpath, f)).read()
                assert not re.search(r"^\s*(import|from)\s+oracle", src, flags=re.M), f


def test_batched_rejects_stream_counts_outside_1_to_32(frt):
    L = frt.lib()
    bad = L.frt_chunk_attention_batched.argtypes[0]._type_
    arr = (bad * 33)()
    for n in (0, -1, 33):
        assert L.frt_chunk_attention_batched(arr, n, arr, arr) == 1, n   # FRT_ERR_INVALID_ARG
        assert "1 <= n <= 32" in L.frt_last_error().decode()
    assert L.frt_chunk_attention_batched(None, 1, arr, arr) == 1


def test_step_group_argument_checks(frt):
    L = frt.lib()
    assert not L.frt_steps_create(0, 2, 64, 16, 3, 3)
    assert not L.frt_steps_create(33, 2, 64, 16, 3, 3)
    assert not L.frt_steps_create(2, 2, 96, 16, 3, 3)      # head_dim unsupported
    g = L.frt_steps_create(3, 2, 64, 16, 3, 3)
    assert g
    assert L.frt_steps_stream(g, 0) and L.frt_steps_stream(g, 2)
    assert not L.frt_steps_stream(g, 3) and not L.frt_steps_stream(g, -1)
    # steps are unconfigured: a tick is a state error, an empty tick is a no-op
    arr = (ctypes.c_void_p * 3)()
    assert L.frt_steps_tick(g, 0, arr, arr, arr, arr) == 0
    assert L.frt_steps_tick(g, 0b1000, arr, arr, arr, arr) == 1
    L.frt_steps_destroy(g)
    L.frt_steps_destroy(None)


def test_gemm_plan_is_host_only_and_checks_arguments(frt):
    # one 128-row tile: a single CTA; two or more: a CTA pair on 256 rows
    assert frt.gemm_plan(128, 1536)[1] == 1
    assert frt.gemm_plan(4680, 1536)[1] == 2
    for M, N, qkv, d in ((4680, 1536, False, 0), (4680, 4608, True, 1536), (300, 200, False, 0)):
        bn, ctas = frt.gemm_plan(M, N, qkv, d)
        assert bn in (128, 192, 256) and ctas in (1, 2)
    # a QKV tile never straddles q, k and v: its width divides d
    assert frt.gemm_plan(4680, 3 * 640, True, 640)[0] == 128
    assert 1536 % frt.gemm_plan(4680, 3 * 1536, True, 1536)[0] == 0
    for args in ((0, 16, False, 0), (16, 0, False, 0), (16, 48, True, 0)):
        with pytest.raises(frt.FrtError):
            frt.gemm_plan(*args)


def _groups(n_q, n_kv, heads):
    """Query groups of one stream in launch order: (KV tiles, one query tile?)."""
    pairs = -(-n_q // 256)
    return [(-(-n_kv // 128), pr * 256 + 128 >= n_q) for _ in range(heads) for pr in range(pairs)]


def _list_schedule(items, sms):
    """Makespan of handing `items` (costs, in order) to the SM that frees first."""
    import heapq
    free = [0.0] * sms
    for c in items:
        t = heapq.heappop(free) + c
        heapq.heappush(free, t)
    return max(free)


def _plan_items(groups, n_full, n_split):
    # the planner's cost model: 7 KV steps per item, 1 more per split item, 0.6 per
    # KV step of a one-tile group
    out = []
    for g, (tiles, single) in enumerate(groups):
        w = 0.6 if single else 1.0
        if g < n_full:
            out.append(7.0 + tiles * w)
        else:
            out += [8.0 + ((s + 1) * tiles // n_split - s * tiles // n_split) * w
                    for s in range(n_split)]
    return out


@pytest.mark.parametrize("n_q,n_kv,heads", [(4680, 32760, 12), (4680, 32760, 40),
                                            (10800, 64800, 40), (4680, 4680, 40),
                                            (256, 5120, 2), (48, 144, 2), (390, 128, 3)])
def test_attention_plan_is_valid_and_beats_whole_and_uniform_splits(frt, n_q, n_kv, heads):
    sms = 152
    n_full, n_split = frt.attention_plan([n_q], [n_kv], heads, sms)
    groups = _groups(n_q, n_kv, heads)
    G = len(groups)
    assert 0 <= n_full <= G and 1 <= n_split <= 4
    if n_split == 1:
        assert n_full == G
    else:
        assert n_full < G
        assert all(t >= 2 * n_split for t, _ in groups[n_full:])   # parts of >= 2 KV tiles
    best = _list_schedule(_plan_items(groups, n_full, n_split), sms)
    assert best <= _list_schedule(_plan_items(groups, G, 1), sms) + 1e-9
    for s in range(2, 5):
        if all(t >= 2 * s for t, _ in groups):
            assert best <= _list_schedule(_plan_items(groups, 0, s), sms) + 1e-9


def test_attention_plan_worked_examples(frt):
    # 1.3B shape: 12 heads x 19 query groups = 228 groups of 256 KV tiles on 152 SMs. One
    # whole wave of 152 groups, then the other 76 cut in two: the second wave is 152
    # halves instead of 76 whole groups next to 76 idle SMs
    assert frt.attention_plan([4680], [32760], 12, 152) == (152, 2)
    # 14B shape: 760 groups = exactly 5 waves: nothing to cut
    assert frt.attention_plan([4680], [32760], 40, 152) == (760, 1)
    # one KV tile per group: nothing can be cut
    assert frt.attention_plan([4680], [100], 12, 152) == (228, 1)
    # two groups on 152 SMs: both cut as finely as allowed
    assert frt.attention_plan([256], [128 * 40], 2, 152) == (0, 4)


def test_attention_plan_checks_arguments(frt):
    with pytest.raises(frt.FrtError):
        frt.attention_plan([0], [10], 2)
    with pytest.raises(frt.FrtError):
        frt.attention_plan([10], [10], 0)


# ---- convolution launch plan (host-only) -------------------------------------------

def _conv_items(total, n_tiles, nhalo, units, split):
    """The kernel's share arithmetic written out: unit u's steps, then its items (tile,
    first halo, end halo) in order."""
    def start(u):
        return u * total // units if split else u * n_tiles // units * nhalo
    out = []
    for u in range(units):
        s, s1 = start(u), start(u + 1)
        while s < s1:
            t = s // nhalo
            ts = t * nhalo
            h0, h1 = s - ts, min(s1, ts + nhalo) - ts
            out.append((u, t, h0, h1, start(u) < ts))
            s = ts + h1
    return out


@pytest.mark.parametrize("n_tiles,nhalo,units", [(42, 18, 76), (78, 9, 76), (126, 18, 152),
                                                 (6, 3, 18), (2, 3, 5), (7, 4, 3), (5, 18, 76),
                                                 (1, 1, 1), (3, 9, 27), (200, 18, 76)])
def test_conv_split_shares_cover_every_step_once_with_distinct_part_slots(n_tiles, nhalo, units):
    total = n_tiles * nhalo
    units = min(units, total)
    items = _conv_items(total, n_tiles, nhalo, units, True)
    seen = [[0] * nhalo for _ in range(n_tiles)]
    slots = {}
    for u, t, h0, h1, last in items:
        assert 0 <= h0 < h1 <= nhalo
        for h in range(h0, h1):
            seen[t][h] += 1
        if (h0, h1) != (0, nhalo):
            # contributors of a split tile: units unit_of(ts) .. unit_of(ts + nhalo - 1)
            first = ((t * nhalo + 1) * units - 1) // total
            lastu = (((t + 1) * nhalo) * units - 1) // total
            assert first <= u <= lastu and lastu > first
            slot = 2 * u + (1 if last else 0)
            assert slot not in slots, "two parts share a workspace slot"
            slots[slot] = (t, u)
    assert all(c == 1 for row in seen for c in row)
    # with every share at least half a tile (the plan's cap on units) a tile has at most
    # three parts: the kernel adds one or two other parts
    if units <= total // ((nhalo + 1) // 2):
        for t in range(n_tiles):
            first = ((t * nhalo + 1) * units - 1) // total
            lastu = (((t + 1) * nhalo) * units - 1) // total
            assert lastu - first + 1 <= 3
    # only a unit's first and last items can be parts of split tiles
    for u in range(units):
        mine = [it for it in items if it[0] == u]
        for k, (_, _, h0, h1, _) in enumerate(mine):
            if 0 < k < len(mine) - 1:
                assert (h0, h1) == (0, nhalo)
    # whole-tile shares cover every tile once
    whole = _conv_items(total, n_tiles, nhalo, min(units, n_tiles), False)
    assert sorted(t for _, t, h0, h1, _ in whole if (h0, h1) == (0, nhalo)) == list(range(n_tiles))
    assert all((h0, h1) == (0, nhalo) for _, _, h0, h1, _ in whole)


def test_conv_plan_worked_examples(frt):
    # 30 x 52 x 384: 42 pixel-tile pairs x 2 tiles of 192 channels = 42 pair tiles of 18
    # halos; whole tiles would leave 34 of 76 SM pairs idle, split gives each pair
    # 756 / 76 = 9.9 halos
    assert frt.conv_plan(384, 384, 3, 3, 3, 30, 52, 3, sms=152) == \
        dict(bn=192, pair=1, units=76, split=1, n_tiles=42, nhalo=18)
    # 60 x 104 x 192: 78 pair tiles on 76 pairs would take two rounds of 9 halos
    assert frt.conv_plan(192, 192, 3, 3, 3, 60, 104, 3, sms=152) == \
        dict(bn=192, pair=1, units=76, split=1, n_tiles=78, nhalo=9)
    # whole tiles only: one round of 126 single-CTA tiles of 128 channels
    assert frt.conv_plan(384, 384, 3, 3, 3, 30, 52, 3, sms=152, split_mode=1) == \
        dict(bn=128, pair=0, units=126, split=0, n_tiles=126, nhalo=18)
    # tiles that fill the units evenly are never split
    p = frt.conv_plan(384, 384, 3, 3, 3, 30, 52, 3, sms=126, bn=128, pair=0)
    assert p["split"] == 0 and p["units"] == 126
    # a forced split of a 2-tile problem: 6 halo steps, at least 2 per unit, so 3 units
    assert frt.conv_plan(64, 256, 3, 3, 3, 9, 17, 1, sms=152, bn=256, pair=1, split_mode=2,
                         units=5) == dict(bn=256, pair=1, units=3, split=1, n_tiles=2, nhalo=3)
    # every plan leaves a tile at most three parts
    for args in [(384, 384, 3, 3, 3, 30, 52, 3), (192, 192, 3, 3, 3, 60, 104, 3),
                 (128, 64, 2, 7, 7, 19, 13, 2), (64, 128, 3, 3, 3, 5, 7, 3)]:
        for sms in (152, 148, 7, 3):
            p = frt.conv_plan(*args, sms=sms, split_mode=2)
            if p["split"]:
                assert p["units"] <= p["n_tiles"] * p["nhalo"] // ((p["nhalo"] + 1) // 2)


def test_conv_plan_checks_arguments(frt):
    with pytest.raises(frt.FrtError):
        frt.conv_plan(48, 64, 3, 3, 3, 8, 8, 2, sms=152)      # Cin not a multiple of 64
    with pytest.raises(frt.FrtError):
        frt.conv_plan(64, 64, 3, 3, 3, 8, 8, 2, sms=152, split_mode=3)
