"""Seeded synthetic inputs shaped like the video world-model workloads.

This module holds workload shapes and random inputs only: none of the
method's arithmetic (no rotation, no cache, no attention). Both the CUDA
path's tests/bench and the oracle-based checks draw their inputs here.

The paper's applications are autoregressive video DiTs (WorldPlay 5B,
LongLive 5B, Krea-Realtime; sections 4.3.2-4.3.4) whose weights and videos
are not available; these synthetic Q/K/V tensors stand in for them. Shapes:
token-major ``[tokens, heads, head_dim]`` bf16, tokens = frames_per_chunk *
grid_h * grid_w (frame chunks, Appendix A.1.1).

Recipe: for workload index ``w``, stream ``s`` and chunk ``c`` a PCG64
generator seeded with SeedSequence([1000*w + s, c]) draws q, k, v (in that
order) as float32 N(0, 1), optionally multiplied per head by a factor drawn
U(0.5, 2) once per stream (SeedSequence([1000*w + s, 999999])), then rounded
to bf16 (round to nearest even). Ragged multi-stream fills are drawn
uniform on {1..W} from SeedSequence([1000*w, 777777]). DiT-block workloads
draw hidden states x ~ N(0, 1) [Nq, heads*head_dim] per chunk and projection
weights ~ N(0, 1/d) once per workload (``chunk_x``, ``block_weights``). Streaming
convolution workloads (``CONV_WORKLOADS``) draw channels-last frames ~ N(0, 1) per chunk
and weights ~ N(0, 1/(taps*Cin)) with a small bias (``conv_chunk``, ``conv_weights``).
"""

from __future__ import annotations

import dataclasses
import math

import numpy as np
import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    index: int               # seed base (1000 * index)
    streams: int
    heads: int
    head_dim: int
    grid_h: int
    grid_w: int
    frames: int              # frames per chunk
    window: int              # window in chunks, counting the current chunk
    chunks: int              # chunks streamed per stream in the full run
    split: tuple             # RoPE head_dim split (d_t, d_h, d_w)
    head_scale: bool = False  # per-head U(0.5, 2) factor on q and k
    ragged_fill: bool = False  # per-stream fill drawn uniform 1..window
    fused_rope: bool = False   # RoPE-Q in the attention prologue
    steps: int = 1             # denoising steps, each with its own KV cache
    block: bool = False        # DiT-block slice: hidden states x and projection weights

    @property
    def tokens_per_frame(self) -> int:
        return self.grid_h * self.grid_w

    @property
    def n_q(self) -> int:
        return self.frames * self.tokens_per_frame

    def n_kv(self, chunk: int) -> int:
        return min(chunk + 1, self.window) * self.n_q

    def attn_flops(self, chunk: int) -> int:
        """4 * Nq * Nkv * D * H: QK^T and PV, one multiply-add = 2 flops."""
        return 4 * self.n_q * self.n_kv(chunk) * self.head_dim * self.heads


WORKLOADS = {
    "tiny": Workload("tiny", 0, 1, 2, 64, 4, 4, 3, 3, 4, (16, 24, 24)),
    "dit1p3b": Workload("dit1p3b", 1, 1, 12, 128, 30, 52, 3, 7, 7, (32, 48, 48)),
    "dit14b": Workload("dit14b", 2, 1, 40, 128, 30, 52, 3, 7, 20, (32, 48, 48),
                       head_scale=True),
    "stream720p": Workload("stream720p", 3, 1, 40, 128, 45, 80, 3, 6, 6,
                           (32, 48, 48), fused_rope=True),
    "multi8": Workload("multi8", 4, 8, 24, 128, 30, 52, 3, 7, 7, (32, 48, 48),
                       ragged_fill=True),
    # four denoising steps of the 1.3B shape, each with its own cache, advanced in
    # pipeline ticks (one batched attention launch per tick)
    "pp4dit1p3b": Workload("pp4dit1p3b", 5, 1, 12, 128, 30, 52, 3, 7, 7, (32, 48, 48),
                           steps=4),
    # the attention slice of a DiT block (QKV projection, RoPE, append, attention,
    # output projection) around the tiny and the 1.3B shapes
    "blocktiny": Workload("blocktiny", 6, 1, 2, 64, 4, 4, 3, 3, 4, (16, 24, 24), block=True),
    "block1p3b": Workload("block1p3b", 7, 1, 12, 128, 30, 52, 3, 7, 7, (32, 48, 48),
                          block=True),
}


def head_scales(wl: Workload, stream: int) -> np.ndarray | None:
    if not wl.head_scale:
        return None
    rng = np.random.Generator(np.random.PCG64(
        np.random.SeedSequence([1000 * wl.index + stream, 999999])))
    return rng.uniform(0.5, 2.0, size=wl.heads).astype(np.float32)


def stream_fills(wl: Workload) -> list[int]:
    """Valid chunks (including the measured one) per stream."""
    if not wl.ragged_fill:
        return [wl.window] * wl.streams
    rng = np.random.Generator(np.random.PCG64(
        np.random.SeedSequence([1000 * wl.index, 777777])))
    return [int(x) for x in rng.integers(1, wl.window + 1, size=wl.streams)]


def random_qkv(n_tokens: int, heads: int, head_dim: int, seed, scales=None):
    """q, k, v bf16 CPU tensors [n_tokens, heads, head_dim] from PCG64(seed)."""
    rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence(seed)))
    out = []
    for which in range(3):
        x = rng.standard_normal((n_tokens, heads, head_dim), dtype=np.float32)
        if scales is not None and which < 2:
            x *= scales[None, :, None]
        out.append(torch.from_numpy(x).to(torch.bfloat16))
    return tuple(out)


def chunk_qkv(wl: Workload, stream: int, chunk: int):
    """Inputs of ``chunk`` of ``stream`` of workload ``wl``."""
    return random_qkv(wl.n_q, wl.heads, wl.head_dim,
                      [1000 * wl.index + stream, chunk], head_scales(wl, stream))


def block_weights(wl: Workload):
    """(w_qkv [3d, d], w_o [d, d]) bf16 CPU tensors, d = heads * head_dim: entries
    N(0, 1/d) (so projections of N(0, 1) hidden states are again about N(0, 1)),
    from PCG64(SeedSequence([1000*w, 555555])), w_qkv drawn first."""
    d = wl.heads * wl.head_dim
    rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence([1000 * wl.index, 555555])))
    sd = np.float32(1.0 / math.sqrt(d))
    w_qkv = rng.standard_normal((3 * d, d), dtype=np.float32) * sd
    w_o = rng.standard_normal((d, d), dtype=np.float32) * sd
    return (torch.from_numpy(w_qkv).to(torch.bfloat16), torch.from_numpy(w_o).to(torch.bfloat16))


def chunk_x(wl: Workload, stream: int, chunk: int) -> torch.Tensor:
    """Hidden states [Nq, d] bf16 of ``chunk``: N(0, 1) from
    PCG64(SeedSequence([1000*w + stream, chunk, 1]))."""
    d = wl.heads * wl.head_dim
    rng = np.random.Generator(np.random.PCG64(
        np.random.SeedSequence([1000 * wl.index + stream, chunk, 1])))
    return torch.from_numpy(rng.standard_normal((wl.n_q, d), dtype=np.float32)).to(torch.bfloat16)


@dataclasses.dataclass(frozen=True)
class ConvWorkload:
    """A streaming causal 3D convolution layer of a video VAE decoder."""
    name: str
    index: int
    cin: int
    cout: int
    kt: int
    kh: int
    kw: int
    grid_h: int
    grid_w: int
    frames: int              # frames per chunk
    chunks: int

    @property
    def taps(self) -> int:
        return self.kt * self.kh * self.kw

    def flops(self) -> int:
        """2 * outputs * Cout * taps * Cin per chunk (one multiply-add = 2 flops)."""
        return 2 * self.frames * self.grid_h * self.grid_w * self.cout * self.taps * self.cin


CONV_WORKLOADS = {
    "convtiny": ConvWorkload("convtiny", 20, 64, 64, 3, 3, 3, 5, 9, 2, 4),
    # decoder layers of a 3-frame chunk: latent grid 30 x 52 at 384 channels, and the
    # 2x upsampled 60 x 104 grid at 192 channels
    "vae30x52c384": ConvWorkload("vae30x52c384", 21, 384, 384, 3, 3, 3, 30, 52, 3, 4),
    "vae60x104c192": ConvWorkload("vae60x104c192", 22, 192, 192, 3, 3, 3, 60, 104, 3, 4),
}


def conv_weights(cw: ConvWorkload):
    """(w [taps, Cout, Cin] bf16, bias [Cout] fp32): w ~ N(0, 1/(taps*Cin)), bias ~
    N(0, 0.1^2), from PCG64(SeedSequence([1000*w, 444444]))."""
    rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence([1000 * cw.index, 444444])))
    sd = np.float32(1.0 / math.sqrt(cw.taps * cw.cin))
    w = rng.standard_normal((cw.taps, cw.cout, cw.cin), dtype=np.float32) * sd
    b = rng.standard_normal(cw.cout, dtype=np.float32) * np.float32(0.1)
    return torch.from_numpy(w).to(torch.bfloat16), torch.from_numpy(b)


def conv_chunk(cw: ConvWorkload, stream: int, chunk: int) -> torch.Tensor:
    """Chunk of input frames [F, H, W, Cin] bf16, N(0, 1), from
    PCG64(SeedSequence([1000*w + stream, chunk, 2]))."""
    rng = np.random.Generator(np.random.PCG64(
        np.random.SeedSequence([1000 * cw.index + stream, chunk, 2])))
    x = rng.standard_normal((cw.frames, cw.grid_h, cw.grid_w, cw.cin), dtype=np.float32)
    return torch.from_numpy(x).to(torch.bfloat16)


def as_f64(t: torch.Tensor) -> np.ndarray:
    """bf16 tensor -> float64 numpy array (exact widening)."""
    return t.detach().to("cpu", torch.float32).numpy().astype(np.float64)


def default_split(head_dim: int) -> tuple:
    """(d_t, d_h, d_w) in the ratio 1/4 : 3/8 : 3/8, each even."""
    d_t = 2 * round(head_dim / 8)
    d_h = 2 * ((head_dim - d_t) // 4)
    return (d_t, d_h, head_dim - d_t - d_h)


def sm_scale(head_dim: int) -> float:
    return 1.0 / math.sqrt(head_dim)
