"""GPU parity of the streaming causal 3D convolution (frt_conv_step) against the fp64
oracle, through the C ABI: every output element at small sizes (ragged against the
16-row x 8-column pixel tiles and their halos), every tile width and pairing the kernel
offers, tiles whose K sum is split over several units (parts added by the last to
arrive), sampled outputs at the VAE-decoder sizes, the frame cache bit-exact,
determinism and the bf16 output.

Tolerance: fp32 accumulation of K = taps * Cin bf16 products, whatever the order, is
within K * 2^-24 * sum |w x| of the exact sum (tested with K * 2^-23 plus 1e-6); a bf16
output adds half an ulp of the result."""

import numpy as np
import pytest
import torch

from oracle.frt_oracle import OracleConvStream, causal_conv3d
from paper_2607_18171_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def frt():
    from paper_2607_18171_gb300 import frt as f
    f.lib()
    return f


def _f64(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def _bound(cw, x_ext, w, out_bf16, ref):
    """Elementwise error bound: K * 2^-23 * (|x_ext| conv |w|) (+ bf16 half ulp)."""
    mag = causal_conv3d(np.abs(x_ext), np.abs(w), np.zeros(cw.cout), cw.kt, cw.kh, cw.kw)
    b = cw.taps * cw.cin * 2.0 ** -23 * mag + 1e-6
    if out_bf16:
        b = b + 2.0 ** -8 * np.abs(ref)
    return b


SMALL = {
    "convtiny": synth.CONV_WORKLOADS["convtiny"],
    # ragged against the tiles, kt = 2 and kh != kw, two k-blocks of channels
    "conv_ragged": synth.ConvWorkload("conv_ragged", 23, 128, 64, 2, 3, 5, 11, 21, 3, 3),
    # one frame per chunk (the cache is shifted, not replaced)
    "conv_f1": synth.ConvWorkload("conv_f1", 24, 64, 256, 3, 3, 3, 9, 17, 1, 4),
    # no temporal taps: nothing cached
    "conv_kt1": synth.ConvWorkload("conv_kt1", 25, 64, 192, 1, 3, 3, 8, 16, 2, 2),
    # an odd number of pixel tiles (3 frames x 1 tile): the last CTA pair has a second
    # half past the chunk, which computes on zero-filled input and stores nothing
    "conv_odd_tiles": synth.ConvWorkload("conv_odd_tiles", 26, 64, 128, 3, 3, 3, 5, 7, 3, 3),
    # a 7 x 7 spatial kernel (halo 14 x 22 pixels), two channel blocks
    "conv_k7": synth.ConvWorkload("conv_k7", 27, 128, 64, 2, 7, 7, 19, 13, 2, 3),
}


@pytest.mark.parametrize("name", list(SMALL))
@pytest.mark.parametrize("out", [torch.float32, torch.bfloat16])
def test_conv_stream_matches_oracle_every_element(frt, name, out):
    _stream_against_oracle(frt, SMALL[name], name, out)


def _stream_against_oracle(frt, cw, name, out, tile=None, split=None):
    w, b = synth.conv_weights(cw)
    wd, bd = w.cuda(), b.cuda()
    st = frt.ConvStream(cw.cin, cw.cout, cw.kt, cw.kh, cw.kw, cw.grid_h, cw.grid_w, cw.frames,
                        out_dtype=out)
    if tile is not None:
        st.set_tile(*tile)
    if split is not None:
        st.set_split(*split)
    outs = []
    orc = OracleConvStream(cw.cin, cw.cout, cw.kt, cw.kh, cw.kw, cw.grid_h, cw.grid_w)
    wf, bf = synth.as_f64(w), b.double().numpy()
    for c in range(cw.chunks):
        x = synth.conv_chunk(cw, 0, c)
        y = st.new_out()
        st.step(x.cuda(), wd, bd, y)
        st.sync()
        x_ext = np.concatenate([orc.cache, synth.as_f64(x)], axis=0)
        ref = orc.step(synth.as_f64(x), wf, bf)
        got = _f64(y)
        outs.append(y)
        bound = _bound(cw, x_ext, wf, out == torch.bfloat16, ref)
        err = np.abs(got - ref)
        assert np.all(err <= bound), f"{name} chunk {c}: max excess {float(np.max(err - bound)):.3e}"
        if cw.kt > 1:
            assert np.array_equal(_f64(st.cache()), orc.cache), f"{name} chunk {c}: cache"
    st.close()
    return outs


# every output-channel tile and pairing the kernel offers, on shapes whose Cout admits
# several of them (Cout 256: 64, 128, 256; Cout 192: 64, 96, 192)
FORCED = [("conv_f1", bn, pr) for bn in (64, 128, 256) for pr in (0, 1)] + \
         [("conv_kt1", bn, pr) for bn in (64, 96, 192) for pr in (0, 1)] + \
         [("conv_odd_tiles", 128, 1), ("conv_ragged", 64, 0)]


@pytest.mark.parametrize("name,bn,pair", FORCED)
def test_conv_every_tile_matches_oracle(frt, name, bn, pair):
    _stream_against_oracle(frt, SMALL[name], f"{name} bn={bn} pair={pair}", torch.float32,
                           tile=(bn, pair))


# tiles split over units (forced): the number of units sets where the parts begin, so
# several counts cover parts of one, two and several halos, a unit holding parts of two
# tiles, and (pairs) both CTAs of a pair adding their own rows
SPLIT = [("conv_f1", 128, 0, 5), ("conv_f1", 256, 1, 5), ("conv_f1", 64, 0, 7),
         ("conv_ragged", 64, 0, 7), ("conv_ragged", 64, 1, 4), ("conv_k7", 64, 1, 3),
         ("conv_k7", 64, 0, 11), ("conv_odd_tiles", 128, 1, 0), ("conv_f1", 0, 0, 0),
         ("convtiny", 0, 0, 0)]


@pytest.mark.parametrize("name,bn,pair,units", SPLIT)
@pytest.mark.parametrize("out", [torch.float32, torch.bfloat16])
def test_conv_split_tiles_match_oracle_every_element(frt, name, bn, pair, units, out):
    if out == torch.bfloat16 and bn % 64:
        pytest.skip("bf16 output needs 64-channel units")
    cw = SMALL[name]
    plan = frt.conv_plan(cw.cin, cw.cout, cw.kt, cw.kh, cw.kw, cw.grid_h, cw.grid_w, cw.frames,
                         torch.cuda.get_device_properties(0).multi_processor_count, out_dtype=out,
                         bn=bn, pair=pair, split_mode=2, units=units)
    assert plan["split"] == 1, plan
    _stream_against_oracle(frt, cw, f"{name} bn={bn} pair={pair} units={units}", out,
                           tile=(bn, pair) if bn else None, split=(2, units))


@pytest.mark.parametrize("mode", [1, 2])
@pytest.mark.parametrize("name,bn,pair,units", [SPLIT[0], SPLIT[1], SPLIT[4], SPLIT[6],
                                                SPLIT[7], SPLIT[9]])
def test_conv_split_tiles_every_gathering_path(frt, name, bn, pair, units, mode):
    """The first part of a split tile gathers the others while its MMAs run when they are
    early; the other paths are forced here: 1 takes every other part only after its own
    accumulator is ready (bulk copies into the idle rings), 2 makes it write itself and
    arrive so that whichever part completes the count adds them all. Both match the
    oracle, and give the bits of the path as built."""
    cw = SMALL[name]
    tile = (bn, pair) if bn else None
    frt.selftest_conv_part_mode(0)
    base = _stream_against_oracle(frt, cw, f"{name} mode 0", torch.float32, tile=tile,
                                  split=(2, units))
    try:
        frt.selftest_conv_part_mode(mode)
        got = _stream_against_oracle(frt, cw, f"{name} mode {mode}", torch.float32, tile=tile,
                                     split=(2, units))
    finally:
        frt.selftest_conv_part_mode(0)
    for c, (a, b) in enumerate(zip(base, got)):
        assert torch.equal(a, b), f"{name}: gathering mode {mode} changed chunk {c}"


def test_conv_split_is_deterministic(frt):
    """Parts are added in step order by whichever part arrives last: the same plan gives
    the same bits on every run."""
    cw = SMALL["conv_k7"]
    w, b = (t.cuda() for t in synth.conv_weights(cw))
    runs = []
    for _ in range(3):
        st = frt.ConvStream(cw.cin, cw.cout, cw.kt, cw.kh, cw.kw, cw.grid_h, cw.grid_w, cw.frames)
        st.set_tile(64, 0)
        st.set_split(2, 11)
        ys = []
        for c in range(cw.chunks):
            y = st.new_out()
            st.step(synth.conv_chunk(cw, 2, c).cuda(), w, b, y)
            ys.append(y)
        st.sync()
        st.close()
        runs.append(ys)
    for other in runs[1:]:
        for a, r in zip(runs[0], other):
            assert torch.equal(a, r)


@pytest.mark.parametrize("name", ["conv_f1", "conv_kt1"])
def test_conv_tile_choice_does_not_change_results(frt, name):
    """With whole tiles each output sums the same products in the same order (temporal
    tap, channel block, spatial tap, 16-channel step) whatever the tile: every choice
    gives the same bits."""
    cw = SMALL[name]
    w, b = (t.cuda() for t in synth.conv_weights(cw))
    results = {}
    for bn in (64, 96, 128, 192, 256):
        if cw.cout % bn:
            continue
        for pr in (0, 1):
            st = frt.ConvStream(cw.cin, cw.cout, cw.kt, cw.kh, cw.kw, cw.grid_h, cw.grid_w,
                                cw.frames)
            st.set_tile(bn, pr)
            st.set_split(1)
            ys = []
            for c in range(cw.chunks):
                y = st.new_out()
                st.step(synth.conv_chunk(cw, 0, c).cuda(), w, b, y)
                ys.append(y)
            st.sync()
            st.close()
            results[(bn, pr)] = ys
    first = next(iter(results.values()))
    for key, ys in results.items():
        for c, (a, r) in enumerate(zip(first, ys)):
            assert torch.equal(a, r), f"{name}: tile {key} differs at chunk {c}"


@pytest.mark.parametrize("name", ["vae30x52c384", "vae60x104c192"])
def test_conv_vae_sizes_on_sampled_pixels(frt, name):
    """Full VAE-decoder sizes: 4 chunks streamed; every output channel of 300 sampled
    pixels (tile edges, frame borders, random) against the oracle's definition."""
    cw = synth.CONV_WORKLOADS[name]
    w, b = synth.conv_weights(cw)
    st = frt.ConvStream(cw.cin, cw.cout, cw.kt, cw.kh, cw.kw, cw.grid_h, cw.grid_w, cw.frames)
    wf, bf = synth.as_f64(w), b.double().numpy()
    rng = np.random.default_rng(5)
    cache = np.zeros((cw.kt - 1, cw.grid_h, cw.grid_w, cw.cin))
    for c in range(cw.chunks):
        x = synth.conv_chunk(cw, 0, c)
        y = st.new_out()
        st.step(x.cuda(), w.cuda(), b.cuda(), y)
        st.sync()
        xf = synth.as_f64(x)
        x_ext = np.concatenate([cache, xf], axis=0)
        got = _f64(y)
        pix = [(t, h, ww) for t in range(cw.frames) for h in (0, 7, 8, 15, 16, cw.grid_h - 1)
               for ww in (0, 7, 8, 15, 16, cw.grid_w - 1)]
        pix += [(int(rng.integers(cw.frames)), int(rng.integers(cw.grid_h)),
                 int(rng.integers(cw.grid_w))) for _ in range(300 - len(pix))]
        ph, pw = cw.kh // 2, cw.kw // 2
        pad = np.zeros((x_ext.shape[0], cw.grid_h + 2 * ph, cw.grid_w + 2 * pw, cw.cin))
        pad[:, ph:ph + cw.grid_h, pw:pw + cw.grid_w] = x_ext
        for (t, h, ww) in pix:
            win = pad[t:t + cw.kt, h:h + cw.kh, ww:ww + cw.kw].reshape(cw.taps, cw.cin)
            ref = bf + np.einsum("koc,kc->o", wf, win)
            mag = np.einsum("koc,kc->o", np.abs(wf), np.abs(win))
            err = np.abs(got[t, h, ww] - ref)
            assert np.all(err <= cw.taps * cw.cin * 2.0 ** -23 * mag + 1e-6), (name, c, t, h, ww)
        cache = x_ext[-(cw.kt - 1):]
        assert np.array_equal(_f64(st.cache()), cache)
    st.close()


def test_conv_is_deterministic_and_reset_restarts(frt):
    cw = SMALL["conv_ragged"]
    w, b = (t.cuda() for t in synth.conv_weights(cw))
    st = frt.ConvStream(cw.cin, cw.cout, cw.kt, cw.kh, cw.kw, cw.grid_h, cw.grid_w, cw.frames)
    runs = []
    for _ in range(2):
        outs = []
        for c in range(3):
            y = st.new_out()
            st.step(synth.conv_chunk(cw, 1, c).cuda(), w, b, y)
            outs.append(y)
        st.sync()
        runs.append(outs)
        st.reset()
    for a, b_ in zip(*runs):
        assert torch.equal(a, b_)
    st.close()


def test_conv_rejects_bad_arguments(frt):
    with pytest.raises(frt.FrtError):
        frt.ConvStream(48, 64, 3, 3, 3, 8, 8, 2)          # Cin not a multiple of 64
    with pytest.raises(frt.FrtError):
        frt.ConvStream(64, 64, 3, 2, 3, 8, 8, 2)          # even kh
    cw = SMALL["convtiny"]
    st = frt.ConvStream(cw.cin, cw.cout, cw.kt, cw.kh, cw.kw, cw.grid_h, cw.grid_w, cw.frames)
    w, b = (t.cuda() for t in synth.conv_weights(cw))
    with pytest.raises(ValueError):
        st.step(torch.zeros(1, 2, 3, 64, dtype=torch.bfloat16, device="cuda"), w, b, st.new_out())
    for bn, pr in ((100, 1), (128, 0), (64, 2)):    # not a width / not dividing Cout / pairing
        with pytest.raises(frt.FrtError):
            st.set_tile(bn, pr)
    for mode, units in ((3, 0), (-1, 0), (2, -1)):
        with pytest.raises(frt.FrtError):
            st.set_split(mode, units)
    st.close()
    # a bf16 output is staged in 64-channel units: a 96-wide tile cannot write it
    cw = SMALL["conv_kt1"]
    st = frt.ConvStream(cw.cin, cw.cout, cw.kt, cw.kh, cw.kw, cw.grid_h, cw.grid_w, cw.frames,
                        out_dtype=torch.bfloat16)
    w, b = (t.cuda() for t in synth.conv_weights(cw))
    st.set_tile(96, 1)
    with pytest.raises(frt.FrtError):
        st.step(synth.conv_chunk(cw, 0, 0).cuda(), w, b, st.new_out())
    st.close()
