"""Shared helpers for the parity tests: run a workload through the C ABI and the
fp64 oracle on the same seeded inputs and compare."""

from __future__ import annotations

import numpy as np
import torch

from oracle.frt_oracle import OracleStream, attention, bf16_round, rope3d
from paper_2607_18171_gb300 import synth

MAX_ABS = 2e-2      # max |err| of fp32 output vs the fp64 oracle
MAX_REL_L2 = 5e-3   # ||err||_2 / ||ref||_2


def compare(gpu_out: np.ndarray, ref: np.ndarray):
    g = np.asarray(gpu_out, dtype=np.float64)
    r = np.asarray(ref, dtype=np.float64)
    err = g - r
    max_abs = float(np.max(np.abs(err)))
    rel = float(np.linalg.norm(err) / max(np.linalg.norm(r), 1e-300))
    return max_abs, rel


def assert_close(gpu_out, ref, what=""):
    max_abs, rel = compare(gpu_out, ref)
    assert np.all(np.isfinite(gpu_out)), f"{what}: non-finite output"
    assert max_abs <= MAX_ABS and rel <= MAX_REL_L2, f"{what}: max|err| {max_abs:.3e} rel-L2 {rel:.3e}"
    return max_abs, rel


def sample_rows(n_q: int, tpf: int, count: int = 256, seed: int = 0) -> np.ndarray:
    """Rows at tile/frame edges and the ragged tail, plus random rows."""
    edges = {0, 1, 127, 128, 255, 256, n_q - 1, n_q - 2, n_q - 129}
    for f in range(1, n_q // tpf + 1):
        edges.update({f * tpf - 1, f * tpf})
    t = (n_q // 128) * 128
    edges.update({t - 1, t})
    edges = {e for e in edges if 0 <= e < n_q}
    rng = np.random.default_rng(seed)
    extra = rng.choice(n_q, size=min(n_q, max(0, count - len(edges))), replace=False)
    return np.array(sorted(edges.union(int(x) for x in extra)), dtype=np.int64)


def oracle_window(wl, stream: int, chunk: int):
    """Rotated (bf16-rounded) K and V of the window ending at `chunk`, and the chunk's
    rotated q, from the oracle (float32 arrays holding bf16 values exactly)."""
    first = max(0, chunk - wl.window + 1)
    ks, vs = [], []
    q_rot = None
    for c in range(first, chunk + 1):
        q, k, v = synth.chunk_qkv(wl, stream, c)
        args = (c, wl.grid_h, wl.grid_w, wl.frames, wl.split)
        ks.append(bf16_round(rope3d(synth.as_f64(k), *args)).astype(np.float32))
        vs.append(synth.as_f64(v).astype(np.float32))
        if c == chunk:
            q_rot = bf16_round(rope3d(synth.as_f64(q), *args)).astype(np.float32)
    return q_rot, np.concatenate(ks), np.concatenate(vs)


def oracle_rows(wl, stream: int, chunk: int, rows):
    q_rot, k, v = oracle_window(wl, stream, chunk)
    return attention(q_rot, k, v, synth.sm_scale(wl.head_dim), rows=rows)


def make_stream(wl, frt, out_dtype=torch.float32):
    return frt.Stream(wl.heads, wl.head_dim, wl.grid_h, wl.grid_w, wl.frames, wl.window,
                      split=wl.split, out_dtype=out_dtype)


def gpu_inputs(wl, stream: int, chunk: int):
    return tuple(t.cuda() for t in synth.chunk_qkv(wl, stream, chunk))


def run_fused(st, wl, stream: int, chunks, keep=()):
    """Stream chunks 0..chunks-1 through frt_chunk_step; return {c: (out, slot, ev)}
    for c in keep."""
    res = {}
    for c in range(chunks):
        q, k, v = gpu_inputs(wl, stream, c)
        out = st.new_out()
        slot, ev = st.chunk_step(q, k, v, out)
        if c in keep:
            res[c] = (out.float().cpu().numpy(), slot, ev)
    st.sync()
    return res


def run_separate(st, wl, stream: int, chunks, keep=()):
    """Same as run_fused through frt_rope3d_qk + frt_kv_append_evict + frt_chunk_attention."""
    res = {}
    for c in range(chunks):
        q, k, v = gpu_inputs(wl, stream, c)
        st.rope3d_qk(q, k)
        slot, ev = st.kv_append_evict(k, v)
        out = st.new_out()
        st.chunk_attention(q, out, k, v)
        if c in keep:
            res[c] = (out.float().cpu().numpy(), slot, ev)
    st.sync()
    return res


def oracle_full_stream(wl, stream: int, chunks: int):
    orc = OracleStream(wl.heads, wl.head_dim, wl.grid_h, wl.grid_w, wl.frames, wl.window,
                       wl.split)
    outs = []
    for c in range(chunks):
        q, k, v = synth.chunk_qkv(wl, stream, c)
        outs.append(orc.step(synth.as_f64(q), synth.as_f64(k), synth.as_f64(v)))
    return outs
