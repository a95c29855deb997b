"""fp64 CPU oracle for streaming frame-chunk attention over a rolling KV cache.

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference legs of ``bench.py`` may import this module. The
product path (``paper_2607_18171_gb300``) never imports it, and this module
imports nothing from the product path: the two share no arithmetic.

What it computes, and where that comes from
-------------------------------------------
The paper (arxiv 2607.18171, "FlashRT") models an autoregressive video DiT
as an operation whose batch ``j`` inherits a persistent KV cache from batch
``j-1`` (section 2, "Problem Formulation": the lambda=1 cross-batch state
edge; Appendix A.1.2 "Pipeline graph": the KV cache shared by batch j+1 and
batch j), with each denoising step owning an independent cache (section 3.1
"Case study"; Appendix A.4). Input arrives as frame chunks (Appendix A.1.1).
The paper gives no formula for the attention itself; the per-chunk
computation below is the plain definition of the workload the paper's video
world models run (sections 4.3.2-4.3.4): 3D rotary position embedding on
Q and K, append of the chunk's K/V to a sliding-window cache, and exact
softmax attention of the chunk's queries over every cached key.

Every function is the plain definition: no online softmax, no tiling, no
fused steps. Library primitives used as steps: ``numpy.matmul`` (dot
products), ``numpy.exp``, ``numpy.cos``/``numpy.sin``.

Readings of points the paper leaves open (each is a convention choice):
  * RoPE pairs are adjacent elements (2j, 2j+1) inside each of the three
    head_dim segments [t | h | w]; pair j of a segment of width d_a turns by
    pos_a * theta**(-2j/d_a), theta = 10000.
  * Positions: t = chunk * frames_per_chunk + frame (absolute frame index
    since stream start), (h, w) = row-major place inside the frame.
  * The window W counts the current chunk: after appending chunk c the cache
    holds chunks max(0, c-W+1) .. c, and chunk c-W is evicted.
  * Every query of the chunk attends every cached key (bidirectional inside
    the chunk, all earlier chunks of the window).
  * Rotated Q and K are rounded to bf16 before attention (they are stored in
    bf16); ``exact=True`` keeps them in fp64 for diagnostics.
"""

from __future__ import annotations

import collections
import math

import numpy as np

__all__ = [
    "bf16_round",
    "token_positions",
    "rope_angles",
    "rope3d",
    "attention",
    "window_index",
    "OracleStream",
]


# ---------------------------------------------------------------------------
# bf16 rounding (IEEE-style round to nearest, ties to even, 8-bit significand)
# ---------------------------------------------------------------------------
def bf16_round(x) -> np.ndarray:
    """Round float64 values to the nearest bfloat16 value (ties to even).

    bfloat16 keeps 8 significant bits (1 implicit + 7 stored) and the float32
    exponent range. For |x| in [2**E, 2**(E+1)) the spacing is 2**(E-7);
    below the smallest normal (2**-126) the spacing stays 2**-133. Values that
    round past the largest finite bf16 become +-inf. The result is returned
    as float64 (every bf16 value is exact in float64).
    """
    x = np.asarray(x, dtype=np.float64)
    out = x.copy()
    nz = np.isfinite(x) & (x != 0.0)
    if not np.any(nz):
        return out
    xv = x[nz]
    _, e = np.frexp(xv)  # xv = m * 2**e, 0.5 <= |m| < 1  ->  leading bit 2**(e-1)
    lead = np.maximum(e - 1, -126)
    ulp = np.ldexp(1.0, lead - 7)
    r = np.rint(xv / ulp) * ulp  # rint: round half to even
    r = np.where(np.abs(r) >= 2.0**128, np.copysign(np.inf, xv), r)
    out[nz] = r
    return out


# ---------------------------------------------------------------------------
# 3D rotary position embedding
# ---------------------------------------------------------------------------
def token_positions(chunk: int, n_tokens: int, grid_h: int, grid_w: int):
    """(t, h, w) position of every token of ``chunk`` (frame-chunk input of
    Appendix A.1.1). Token i of the chunk is frame f = i // (grid_h*grid_w),
    row r = (i mod grid_h*grid_w) // grid_w, column i mod grid_w. The returned
    t is the within-chunk frame f; the caller adds chunk * frames_per_chunk.
    """
    tpf = grid_h * grid_w
    i = np.arange(n_tokens, dtype=np.int64)
    f = i // tpf
    r = (i % tpf) // grid_w
    col = i % grid_w
    return f, r, col


def rope_angles(pos: np.ndarray, width: int, theta: float) -> np.ndarray:
    """Angle of pair j at integer position ``pos`` in a segment of ``width``
    dims: pos * theta**(-2j/width), j = 0 .. width/2 - 1. Shape [len(pos), width/2]."""
    j = np.arange(width // 2, dtype=np.float64)
    inv_freq = np.power(float(theta), -2.0 * j / float(width))
    return np.outer(np.asarray(pos, dtype=np.float64), inv_freq)


def rope3d(x: np.ndarray, chunk: int, grid_h: int, grid_w: int,
           frames_per_chunk: int, split, theta: float = 10000.0) -> np.ndarray:
    """Return a rotated float64 copy of ``x`` ([tokens, heads, head_dim]).

    head_dim is cut into segments [d_t | d_h | d_w] (``split``); in segment a
    the pair (x[o+2j], x[o+2j+1]) turns by angle phi = pos_a * theta**(-2j/d_a):
    (x0, x1) -> (x0 cos phi - x1 sin phi, x0 sin phi + x1 cos phi).
    """
    x = np.asarray(x, dtype=np.float64)
    n_tok, _, dim = x.shape
    d_t, d_h, d_w = (int(s) for s in split)
    if d_t + d_h + d_w != dim or d_t % 2 or d_h % 2 or d_w % 2:
        raise ValueError("rope split must be even and sum to head_dim")
    f, r, col = token_positions(chunk, n_tok, grid_h, grid_w)
    t = chunk * frames_per_chunk + f
    out = x.copy()
    offset = 0
    for pos, width in ((t, d_t), (r, d_h), (col, d_w)):
        if width:
            ang = rope_angles(pos, width, theta)[:, None, :]  # [tok, 1, width/2]
            c, s = np.cos(ang), np.sin(ang)
            x0 = x[:, :, offset + 0: offset + width: 2]
            x1 = x[:, :, offset + 1: offset + width: 2]
            out[:, :, offset + 0: offset + width: 2] = x0 * c - x1 * s
            out[:, :, offset + 1: offset + width: 2] = x0 * s + x1 * c
        offset += width
    return out


# ---------------------------------------------------------------------------
# Exact softmax attention (plain definition)
# ---------------------------------------------------------------------------
def attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, scale: float,
              rows=None, return_probs: bool = False, row_block: int = 512):
    """O[i,h,:] = sum_j softmax_j(scale * <q[i,h], k[j,h]>) v[j,h,:].

    q: [Nq, H, D]; k, v: [Nkv, H, D] (float64). ``rows`` selects a subset of
    query rows (sampled parity); ``None`` means all. Rows are independent, so
    they are evaluated ``row_block`` at a time only to bound memory.
    Returns out [len(rows), H, D] (and the probabilities [len(rows), H, Nkv]
    when ``return_probs``).
    """
    rows = np.arange(q.shape[0]) if rows is None else np.asarray(rows, dtype=np.int64)
    n_heads = q.shape[1]
    out = np.empty((len(rows), n_heads, v.shape[2]), dtype=np.float64)
    probs = np.empty((len(rows), n_heads, k.shape[0])) if return_probs else None
    for h in range(n_heads):
        # widen one head at a time (inputs may be float32 holding bf16 values exactly)
        kh = np.asarray(k[:, h, :], dtype=np.float64)
        vh = np.asarray(v[:, h, :], dtype=np.float64)
        for b0 in range(0, len(rows), row_block):
            rb = rows[b0: b0 + row_block]
            qh = np.asarray(q[rb, h, :], dtype=np.float64)
            scores = scale * (qh @ kh.T)                    # [rows, Nkv]
            m = scores.max(axis=1, keepdims=True)
            e = np.exp(scores - m)
            p = e / e.sum(axis=1, keepdims=True)
            out[b0: b0 + len(rb), h, :] = p @ vh
            if return_probs:
                probs[b0: b0 + len(rb), h, :] = p
    return (out, probs) if return_probs else out


# ---------------------------------------------------------------------------
# Sliding-window cache indices
# ---------------------------------------------------------------------------
def window_index(chunk: int, window: int):
    """Ring slot written by ``chunk``, the chunk it evicts (-1 if none) and the
    number of valid chunks after the append (window counts the current chunk)."""
    if chunk < 0 or window < 1:
        raise ValueError("chunk >= 0 and window >= 1 required")
    slot = chunk % window
    evicted = chunk - window if chunk >= window else -1
    valid = min(chunk + 1, window)
    return slot, evicted, valid


class OracleStream:
    """One stream's persistent state: a deque of the last W chunks of
    (rotated K, V), i.e. the cross-batch KV-cache state edge of section 2.

    ``step(q, k, v)`` runs one frame chunk: RoPE on q and k, append with
    eviction, attention of the chunk's queries over the whole window.
    """

    def __init__(self, heads: int, head_dim: int, grid_h: int, grid_w: int,
                 frames_per_chunk: int, window_chunks: int, split,
                 theta: float = 10000.0, scale: float | None = None,
                 exact: bool = False):
        self.heads = heads
        self.head_dim = head_dim
        self.grid_h = grid_h
        self.grid_w = grid_w
        self.frames_per_chunk = frames_per_chunk
        self.window = window_chunks
        self.split = tuple(int(s) for s in split)
        self.theta = float(theta)
        self.scale = 1.0 / math.sqrt(head_dim) if scale is None else float(scale)
        self.exact = exact
        self.n_q = frames_per_chunk * grid_h * grid_w
        self.chunk = 0
        self.cache = collections.deque()  # entries: (chunk index, k_rot, v)

    def rope(self, q, k):
        """Rotate q and k at the current chunk's positions; round to bf16
        unless ``exact``."""
        args = (self.chunk, self.grid_h, self.grid_w, self.frames_per_chunk,
                self.split, self.theta)
        q_r = rope3d(q, *args)
        k_r = rope3d(k, *args)
        if not self.exact:
            q_r, k_r = bf16_round(q_r), bf16_round(k_r)
        return q_r, k_r

    def append(self, k_rot, v):
        """Append chunk ``self.chunk``; evict the chunk that leaves the window."""
        slot, evicted, _ = window_index(self.chunk, self.window)
        self.cache.append((self.chunk, np.asarray(k_rot, np.float64),
                           np.asarray(v, np.float64)))
        if len(self.cache) > self.window:
            gone, _, _ = self.cache.popleft()
            assert gone == evicted
        self.chunk += 1
        return slot, evicted

    def cached_kv(self):
        """Concatenation of every valid cached chunk's K and V, oldest first."""
        k = np.concatenate([e[1] for e in self.cache], axis=0)
        v = np.concatenate([e[2] for e in self.cache], axis=0)
        return k, v

    def attend(self, q_rot, rows=None, return_probs=False):
        k, v = self.cached_kv()
        return attention(q_rot, k, v, self.scale, rows=rows,
                         return_probs=return_probs)

    def step(self, q, k, v, rows=None):
        """One frame chunk: (out, slot, evicted)."""
        q_r, k_r = self.rope(q, k)
        slot, evicted = self.append(k_r, v)
        return self.attend(q_r, rows=rows), slot, evicted


def linear(x, w) -> np.ndarray:
    """A linear layer without bias in fp64: ``x`` [tokens, in_features], ``w``
    [out_features, in_features]; output feature j of a token is the dot product
    of the token's features with row j of ``w``."""
    return np.asarray(x, np.float64) @ np.asarray(w, np.float64).T


class OracleBlock:
    """The attention slice of one DiT block over a stream: QKV projection, the
    chunk step of ``OracleStream`` (RoPE, append/evict, attention), output
    projection. The paper's video pipelines run their per-chunk attention inside
    such blocks (section 4.2); it gives no formula for them.

    Readings (the paper is silent): ``w_qkv`` [3d, d] stacks the q, k and v
    projections in that order (d = heads * head_dim, each output token-major
    [tokens, heads, head_dim]); no bias and no normalisation; the projection
    output is rounded to bf16 (q, k, v are bf16 tensors on the whole path) before
    RoPE, and the attention output is rounded to bf16 before the output
    projection ``w_o`` [d, d].
    """

    def __init__(self, w_qkv, w_o, heads: int, head_dim: int, grid_h: int, grid_w: int,
                 frames_per_chunk: int, window_chunks: int, split, theta: float = 10000.0):
        self.d = heads * head_dim
        self.w_qkv = np.asarray(w_qkv, np.float64)
        self.w_o = np.asarray(w_o, np.float64)
        assert self.w_qkv.shape == (3 * self.d, self.d) and self.w_o.shape == (self.d, self.d)
        self.stream = OracleStream(heads, head_dim, grid_h, grid_w, frames_per_chunk,
                                   window_chunks, split, theta)

    def project_qkv(self, x):
        """(q, k, v), each [tokens, heads, head_dim], bf16-rounded projections of x."""
        s = self.stream
        qkv = bf16_round(linear(x, self.w_qkv))
        n = qkv.shape[0]
        return tuple(qkv[:, i * self.d:(i + 1) * self.d].reshape(n, s.heads, s.head_dim)
                     for i in range(3))

    def step(self, x, rows=None) -> dict:
        """One frame chunk of hidden states x [Nq, d]. Returns the rotated q and k,
        v, the attention output o and the block output y (o and y for ``rows``
        only, if given), and the append's slot / evicted chunk."""
        q, k, v = self.project_qkv(x)
        q_r, k_r = self.stream.rope(q, k)
        slot, evicted = self.stream.append(k_r, v)
        o = self.stream.attend(q_r, rows=rows)
        y = linear(bf16_round(o).reshape(o.shape[0], self.d), self.w_o)
        return {"q_rot": q_r, "k_rot": k_r, "v": v, "o": o, "y": y, "slot": slot,
                "evicted": evicted}


def causal_conv3d(x_ext, w, bias, kt: int, kh: int, kw: int) -> np.ndarray:
    """Causal 3D convolution of channels-last frames in fp64.

    ``x_ext`` [kt - 1 + F, H, W, Cin]: the kt - 1 frames before the chunk followed by the
    chunk's F frames; ``w`` [kt * kh * kw, Cout, Cin] with tap index (dt * kh + dh) * kw
    + dw; ``bias`` [Cout]. Output frame t (0..F-1) at (h, w):
        y[t, h, w, o] = bias[o] + sum over dt, dh, dw, c of
                        w[tap, o, c] * x_ext[t + dt, h + dh - kh // 2, w + dw - kw // 2, c],
    with positions outside the frame read as zero (spatial zero padding, stride 1)."""
    x_ext = np.asarray(x_ext, np.float64)
    w = np.asarray(w, np.float64)
    n_ext, H, W, cin = x_ext.shape
    F = n_ext - (kt - 1)
    cout = w.shape[1]
    ph, pw = kh // 2, kw // 2
    padded = np.zeros((n_ext, H + 2 * ph, W + 2 * pw, cin))
    padded[:, ph:ph + H, pw:pw + W, :] = x_ext
    y = np.broadcast_to(np.asarray(bias, np.float64), (F, H, W, cout)).copy()
    for dt in range(kt):
        for dh in range(kh):
            for dw in range(kw):
                tap = (dt * kh + dh) * kw + dw
                win = padded[dt:dt + F, dh:dh + H, dw:dw + W, :]
                y += win @ w[tap].T
    return y


class OracleConvStream:
    """A streaming causal 3D convolution layer: the per-stream state is the last kt - 1
    input frames (zeros before the first chunk), the kind of recurrent state a streaming
    video VAE decoder carries from one batch to the next (the (V, V, 1) self-edge of the
    DiT -> VAE pipeline, App. A.3)."""

    def __init__(self, cin: int, cout: int, kt: int, kh: int, kw: int, grid_h: int,
                 grid_w: int):
        self.kt, self.kh, self.kw = kt, kh, kw
        self.cache = np.zeros((kt - 1, grid_h, grid_w, cin))

    def step(self, x, w, bias):
        """One chunk of frames x [F, H, W, Cin]: output [F, H, W, Cout]; the cache then
        holds the last kt - 1 frames of (cache, x)."""
        x = np.asarray(x, np.float64)
        x_ext = np.concatenate([self.cache, x], axis=0)
        y = causal_conv3d(x_ext, w, bias, self.kt, self.kh, self.kw)
        if self.kt > 1:
            self.cache = x_ext[-(self.kt - 1):].copy()
        return y
