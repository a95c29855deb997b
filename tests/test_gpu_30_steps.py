"""Per-denoising-step caches (each step owns its KV cache; step i of chunk c+1 depends
only on step i of chunk c): a wavefront of pipeline ticks, each one batched attention
launch over the active steps, must reproduce every step's own oracle stream."""

import numpy as np
import pytest
import torch

from oracle.frt_oracle import OracleStream
from paper_2607_18171_gb300 import synth
from tests import parity_util as U

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def frt():
    from paper_2607_18171_gb300 import frt as m
    m.lib()
    return m


@pytest.mark.parametrize("n_steps,window,chunks", [(3, 3, 5), (4, 2, 3), (32, 2, 2)])
def test_wavefront_ticks_match_per_step_oracles(frt, n_steps, window, chunks):
    base = synth.Workload("steps", 96, 1, 3, 128, 10, 13, 3, window, chunks, (32, 48, 48))
    grp = frt.Steps(n_steps, base.heads, base.head_dim, base.grid_h, base.grid_w, base.frames,
                    base.window, split=base.split)
    orcs = [OracleStream(base.heads, base.head_dim, base.grid_h, base.grid_w, base.frames,
                         base.window, base.split) for _ in range(n_steps)]
    got, keep = {}, []
    for t in range(chunks + n_steps - 1):
        active = [i for i in range(n_steps) if 0 <= t - i < chunks]
        q, k, v, out = {}, {}, {}, {}
        for i in active:
            q[i], k[i], v[i] = U.gpu_inputs(base, i, t - i)   # step i's own inputs
            out[i] = torch.empty(grp.shape(), dtype=torch.float32, device="cuda")
            got[(i, t - i)] = out[i]
        keep.append((q, k, v))
        grp.tick(active, q, k, v, out)
    grp.sync()
    for i in range(n_steps):
        assert grp.counter(i) == chunks
        for c in range(chunks):
            qh, kh, vh = synth.chunk_qkv(base, i, c)
            ref = orcs[i].step(synth.as_f64(qh), synth.as_f64(kh), synth.as_f64(vh))[0]
            U.assert_close(got[(i, c)].cpu().numpy(), ref, f"step {i} chunk {c}")
    grp.close()
