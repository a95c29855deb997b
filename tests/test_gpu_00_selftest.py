"""Building blocks of the attention kernel, each checked in isolation on the GPU:
a 128x128x128 bf16 tile through TMA + tcgen05.mma (both B layouts, A from shared
memory or TMEM), and the bounded-wait timeout path."""

import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def frt():
    from paper_2607_18171_gb300 import frt as m
    m.lib()
    return m


def _ab(seed):
    g = torch.Generator().manual_seed(seed)
    a = torch.randn(128, 128, generator=g).to(torch.bfloat16)
    b = torch.randn(128, 128, generator=g).to(torch.bfloat16)
    return a, b


def _check(c, ref):
    err = (c.cpu().double() - ref).abs().max().item()
    assert err < 1e-3 * max(1.0, ref.abs().max().item()), err


def test_umma_tile_b_k_major(frt):
    a, b = _ab(1)
    c = frt.selftest_umma_tile(a.cuda(), b.cuda(), b_mn_major=False)
    _check(c, a.double() @ b.double().T)


def test_umma_tile_b_mn_major(frt):
    a, b = _ab(2)
    c = frt.selftest_umma_tile(a.cuda(), b.cuda(), b_mn_major=True, lbo=16384, sbo=1024)
    _check(c, a.double() @ b.double())


def test_umma_tile_a_from_tmem(frt):
    a, b = _ab(3)
    c = frt.selftest_umma_tile(a.cuda(), b.cuda(), b_mn_major=True, lbo=16384, sbo=1024,
                               a_from_tmem=True)
    _check(c, a.double() @ b.double())


def test_bounded_wait_reports_timeout_and_context_survives(frt):
    from paper_2607_18171_gb300 import synth
    wl = synth.WORKLOADS["tiny"]
    st = frt.Stream(wl.heads, wl.head_dim, wl.grid_h, wl.grid_w, wl.frames, wl.window,
                    split=wl.split)
    frt.selftest_wait_timeout(st, 10_000_000)  # 10 ms, nothing ever arrives
    with pytest.raises(frt.FrtError) as ei:
        st.sync()
    assert ei.value.status == 6
    # the status is sticky until reset; the context keeps working
    q, k, v = (t.cuda() for t in synth.chunk_qkv(wl, 0, 0))
    with pytest.raises(frt.FrtError):
        st.chunk_step(q, k, v, st.new_out())
    st.reset()
    out = st.new_out()
    st.chunk_step(q, k, v, out)
    st.sync()
    assert torch.isfinite(out).all()
    st.close()


def test_umma_cta_pair_tile(frt):
    """tcgen05.mma.cta_group::2 on a CTA pair: A rows split across the CTAs, B split by N."""
    g = torch.Generator().manual_seed(4)
    a = torch.randn(256, 128, generator=g).to(torch.bfloat16)
    b = torch.randn(128, 128, generator=g).to(torch.bfloat16)
    c, taddrs = frt.selftest_umma_pair(a.cuda(), b.cuda())
    assert taddrs[0] == taddrs[1]      # one allocation shared by the pair
    _check(c, a.double() @ b.double().T)


def test_umma_cta_pair_pv_tile(frt):
    """The attention's P.V product on a CTA pair: A (P) from TMEM, B (V) MN-major and
    split by its N columns (head_dim halves) across the two CTAs."""
    g = torch.Generator().manual_seed(5)
    a = torch.randn(256, 128, generator=g).to(torch.bfloat16)
    b = torch.randn(128, 128, generator=g).to(torch.bfloat16)
    c, taddrs = frt.selftest_umma_pair(a.cuda(), b.cuda(), pv=True)
    assert taddrs[0] == taddrs[1]
    _check(c, a.double() @ b.double())
