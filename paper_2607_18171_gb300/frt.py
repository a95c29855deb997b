"""Thin ctypes binding of ``libfrt.so`` (C ABI in ``include/frt.h``).

Argument marshalling only: tensors are passed as raw device pointers and every step
of the path runs in the library's CUDA kernels. There is no CPU fallback: if the
library is missing, loading raises.
"""

from __future__ import annotations

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
# FRT_LIBRARY=debug loads the FRT_DEBUG build (bounds-checking kernels, guard words checked
# at every sync); built by _build.build(debug=True)
LIB_PATH = os.path.join(_HERE, "libfrt_debug.so" if os.environ.get("FRT_LIBRARY") == "debug"
                        else "libfrt.so")

FRT_OK = 0
STATUS_NAMES = {0: "FRT_OK", 1: "FRT_ERR_INVALID_ARG", 2: "FRT_ERR_STATE", 3: "FRT_ERR_OOM",
                4: "FRT_ERR_CUDA", 5: "FRT_ERR_UNSUPPORTED", 6: "FRT_ERR_TIMEOUT",
                7: "FRT_ERR_BOUNDS"}
OUT_F32, OUT_BF16 = 0, 1


class FrtError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


class Config(ctypes.Structure):
    _fields_ = [("grid_h", ctypes.c_int), ("grid_w", ctypes.c_int),
                ("rope_dt", ctypes.c_int), ("rope_dh", ctypes.c_int), ("rope_dw", ctypes.c_int),
                ("theta", ctypes.c_double), ("sm_scale", ctypes.c_double),
                ("out_dtype", ctypes.c_int), ("cuda_stream", ctypes.c_void_p)]


_lib = None


def lib() -> ctypes.CDLL:
    """Load libfrt.so once and declare its signatures."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is not built; run __graft_entry__.build() "
                           "(this package has no CPU fallback)")
    L = ctypes.CDLL(LIB_PATH)
    P, I, LL, D = ctypes.c_void_p, ctypes.c_int, ctypes.c_longlong, ctypes.c_double
    sig = {
        "frt_stream_create": (P, [I, I, I, I, I]),
        "frt_config_default": (I, [P, ctypes.POINTER(Config)]),
        "frt_stream_configure": (I, [P, ctypes.POINTER(Config)]),
        "frt_rope3d_qk": (I, [P, P, P]),
        "frt_kv_append_evict": (I, [P, P, P, ctypes.POINTER(I), ctypes.POINTER(LL)]),
        "frt_chunk_attention": (I, [P, P, P, P, P]),
        "frt_chunk_step": (I, [P, P, P, P, P, ctypes.POINTER(I), ctypes.POINTER(LL)]),
        "frt_chunk_step_host": (I, [P, P, P, P, P, ctypes.POINTER(I), ctypes.POINTER(LL)]),
        "frt_chunk_attention_batched": (I, [ctypes.POINTER(P), I, ctypes.POINTER(P),
                                            ctypes.POINTER(P)]),
        "frt_stream_sync": (I, [P]),
        "frt_stream_reset": (I, [P]),
        "frt_stream_destroy": (None, [P]),
        "frt_stream_chunk_counter": (LL, [P]),
        "frt_stream_cache": (I, [P, ctypes.POINTER(P), ctypes.POINTER(P), ctypes.POINTER(LL)]),
        "frt_stream_save": (I, [P, P, P, ctypes.POINTER(LL)]),
        "frt_stream_restore": (I, [P, P, P, LL]),
        "frt_stream_check_guards": (I, [P]),
        "frt_debug_build": (I, []),
        "frt_selftest_append_past_ring": (I, []),
        "frt_selftest_poke_guard": (I, [P, I]),
        "frt_stream_set_attention_events": (I, [P, P, P]),
        "frt_stream_set_append_events": (I, [P, P, P]),
        "frt_chunk_attention_noalloc": (I, [P, P, P, P, I, I, I, I, D, I, P, P]),
        "frt_block_step": (I, [P, P, P, P, P, P, P, ctypes.POINTER(I), ctypes.POINTER(LL)]),
        "frt_conv_create": (P, [I, I, I, I, I, I, I, I]),
        "frt_conv_configure": (I, [P, I, P]),
        "frt_conv_step": (I, [P, P, P, P, P]),
        "frt_conv_cache": (I, [P, ctypes.POINTER(P)]),
        "frt_conv_set_tile": (I, [P, I, I]),
        "frt_conv_set_split": (I, [P, I, I]),
        "frt_conv_plan": (I, [I, I, I, I, I, I, I, I, I, I, I, I, I, I, ctypes.POINTER(ctypes.c_int)]),
        "frt_conv_sync": (I, [P]),
        "frt_conv_reset": (I, [P]),
        "frt_conv_destroy": (None, [P]),
        "frt_gemm_bf16": (I, [P, P, P, I, I, I, I, I, P, P]),
        "frt_gemm_plan": (I, [I, I, I, I, ctypes.POINTER(I), ctypes.POINTER(I)]),
        "frt_attention_plan": (I, [I, ctypes.POINTER(I), ctypes.POINTER(LL), I, I,
                                   ctypes.POINTER(I), ctypes.POINTER(I)]),
        "frt_stream_set_block_events": (I, [P, P, P, P, P]),
        "frt_window_index": (I, [LL, I, ctypes.POINTER(I), ctypes.POINTER(LL),
                                 ctypes.POINTER(I)]),
        "frt_status_string": (ctypes.c_char_p, [I]),
        "frt_last_error": (ctypes.c_char_p, []),
        "frt_version": (ctypes.c_char_p, []),
        "frt_selftest_umma_tile": (I, [P, P, P, I, I, I, I, P, P]),
        "frt_selftest_wait_timeout": (I, [P, LL, P]),
        "frt_selftest_umma_pair": (I, [P, P, P, P, P, P]),
        "frt_selftest_umma_pair_pv": (I, [P, P, P, P, P, P]),
        "frt_selftest_gemm_force_bn": (I, [I]),
        "frt_selftest_conv_part_mode": (I, [I]),
        "frt_steps_create": (P, [I, I, I, I, I, I]),
        "frt_steps_configure": (I, [P, ctypes.POINTER(Config)]),
        "frt_steps_stream": (P, [P, I]),
        "frt_steps_tick": (I, [P, ctypes.c_uint, ctypes.POINTER(P), ctypes.POINTER(P),
                               ctypes.POINTER(P), ctypes.POINTER(P)]),
        "frt_steps_destroy": (None, [P]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(L, name)
        fn.restype = res
        fn.argtypes = args
    _lib = L
    return L


def _check(status: int) -> None:
    if status != FRT_OK:
        raise FrtError(status, lib().frt_last_error().decode())


def _ptr(t: torch.Tensor | None):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _bf16_dev(t: torch.Tensor, shape, name: str) -> None:
    if t.dtype != torch.bfloat16 or not t.is_cuda or not t.is_contiguous():
        raise ValueError(f"{name} must be a contiguous bf16 CUDA tensor")
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")


def window_index(chunk: int, window: int):
    """(slot, evicted, valid_chunks) computed by the library (host only)."""
    s, v = ctypes.c_int(), ctypes.c_int()
    e = ctypes.c_longlong()
    _check(lib().frt_window_index(chunk, window, ctypes.byref(s), ctypes.byref(e),
                                  ctypes.byref(v)))
    return s.value, e.value, v.value


class Stream:
    """One stream's persistent state (its rolling KV cache) on the current device."""

    def __init__(self, heads: int, head_dim: int, grid_h: int, grid_w: int,
                 frames_per_chunk: int, window_chunks: int, split=None, theta: float = 10000.0,
                 sm_scale: float = 0.0, out_dtype: torch.dtype = torch.float32,
                 cuda_stream: torch.cuda.Stream | None = None):
        L = lib()
        self._h = L.frt_stream_create(heads, head_dim, grid_h * grid_w, frames_per_chunk,
                                      window_chunks)
        if not self._h:
            raise FrtError(1, L.frt_last_error().decode())
        self.heads, self.head_dim = heads, head_dim
        self.grid_h, self.grid_w = grid_h, grid_w
        self.frames, self.window = frames_per_chunk, window_chunks
        self.n_q = frames_per_chunk * grid_h * grid_w
        self.out_dtype = out_dtype
        cfg = Config()
        _check(L.frt_config_default(self._h, ctypes.byref(cfg)))
        cfg.grid_h, cfg.grid_w = grid_h, grid_w
        if split is not None:
            cfg.rope_dt, cfg.rope_dh, cfg.rope_dw = (int(x) for x in split)
        cfg.theta = theta
        cfg.sm_scale = sm_scale
        cfg.out_dtype = OUT_BF16 if out_dtype == torch.bfloat16 else OUT_F32
        self.torch_stream = cuda_stream or torch.cuda.current_stream()
        cfg.cuda_stream = ctypes.c_void_p(self.torch_stream.cuda_stream)
        self.config = cfg
        _check(L.frt_stream_configure(self._h, ctypes.byref(cfg)))

    # -- lifetime --------------------------------------------------------------------
    def close(self) -> None:
        if getattr(self, "_h", None):
            h, self._h = self._h, None
            # the debug build compares the cache's guard words before every release
            rc = lib().frt_stream_check_guards(h) if lib().frt_debug_build() else FRT_OK
            msg = lib().frt_last_error().decode() if rc != FRT_OK else ""
            lib().frt_stream_destroy(h)
            if rc not in (FRT_OK, 2):   # 2: never configured
                raise FrtError(rc, msg)

    def __del__(self):  # pragma: no cover - best effort
        try:
            self.close()
        except Exception:
            pass

    @property
    def handle(self):
        return self._h

    @property
    def counter(self) -> int:
        return lib().frt_stream_chunk_counter(self._h)

    def shape(self):
        return (self.n_q, self.heads, self.head_dim)

    def new_out(self) -> torch.Tensor:
        return torch.empty(self.shape(), dtype=self.out_dtype, device="cuda")

    # -- the three operations ------------------------------------------------------
    def rope3d_qk(self, q: torch.Tensor, k: torch.Tensor) -> None:
        _bf16_dev(q, self.shape(), "q"); _bf16_dev(k, self.shape(), "k")
        _check(lib().frt_rope3d_qk(self._h, _ptr(q), _ptr(k)))

    def kv_append_evict(self, k: torch.Tensor, v: torch.Tensor):
        _bf16_dev(k, self.shape(), "k"); _bf16_dev(v, self.shape(), "v")
        slot, ev = ctypes.c_int(), ctypes.c_longlong()
        _check(lib().frt_kv_append_evict(self._h, _ptr(k), _ptr(v), ctypes.byref(slot),
                                         ctypes.byref(ev)))
        return slot.value, ev.value

    def chunk_attention(self, q: torch.Tensor, out: torch.Tensor, k=None, v=None) -> None:
        _bf16_dev(q, self.shape(), "q")
        self._check_out(out)
        _check(lib().frt_chunk_attention(_ptr(q), _ptr(k), _ptr(v), _ptr(out), self._h))

    def chunk_step(self, q, k, v, out):
        for t, n in ((q, "q"), (k, "k"), (v, "v")):
            _bf16_dev(t, self.shape(), n)
        self._check_out(out)
        slot, ev = ctypes.c_int(), ctypes.c_longlong()
        _check(lib().frt_chunk_step(self._h, _ptr(q), _ptr(k), _ptr(v), _ptr(out),
                                    ctypes.byref(slot), ctypes.byref(ev)))
        return slot.value, ev.value

    def chunk_step_host(self, q_host, k_host, v_host, out_host):
        """Host tensors in, host tensor out (copies enqueued on the stream)."""
        for t in (q_host, k_host, v_host, out_host):
            if t.is_cuda or not t.is_contiguous():
                raise ValueError("host buffers must be contiguous CPU tensors")
        slot, ev = ctypes.c_int(), ctypes.c_longlong()
        _check(lib().frt_chunk_step_host(self._h, _ptr(q_host), _ptr(k_host), _ptr(v_host),
                                         _ptr(out_host), ctypes.byref(slot), ctypes.byref(ev)))
        return slot.value, ev.value

    def block_step(self, x, w_qkv, w_o, q_buf, o_buf, y):
        """DiT-block attention slice of the next chunk: x [Nq, d] -> y [Nq, d]
        (d = heads * head_dim); q_buf / o_buf are [Nq, d] bf16 work buffers."""
        n_q = self.shape()[0]
        d = self.heads * self.head_dim
        _bf16_dev(x, (n_q, d), "x")
        _bf16_dev(w_qkv, (3 * d, d), "w_qkv")
        _bf16_dev(w_o, (d, d), "w_o")
        _bf16_dev(q_buf, (n_q, d), "q_buf")
        _bf16_dev(o_buf, (n_q, d), "o_buf")
        if y.dtype != self.out_dtype or not y.is_cuda or not y.is_contiguous() or \
                tuple(y.shape) != (n_q, d):
            raise ValueError("y must be a contiguous [Nq, d] CUDA tensor of the stream's out dtype")
        slot, ev = ctypes.c_int(), ctypes.c_longlong()
        _check(lib().frt_block_step(self._h, _ptr(x), _ptr(w_qkv), _ptr(w_o), _ptr(q_buf),
                                    _ptr(o_buf), _ptr(y), ctypes.byref(slot), ctypes.byref(ev)))
        return slot.value, ev.value

    def set_block_events(self, qkv_start=None, qkv_stop=None, out_start=None, out_stop=None):
        """Record events around the two projection launches of block_step."""
        ev = [None if e is None else ctypes.c_void_p(e.cuda_event)
              for e in (qkv_start, qkv_stop, out_start, out_stop)]
        _check(lib().frt_stream_set_block_events(self._h, *ev))

    def sync(self) -> None:
        _check(lib().frt_stream_sync(self._h))

    def reset(self) -> None:
        _check(lib().frt_stream_reset(self._h))

    def set_attention_events(self, start: torch.cuda.Event | None,
                             stop: torch.cuda.Event | None) -> None:
        """Record these events around every attention kernel launch of this stream."""
        _check(lib().frt_stream_set_attention_events(
            self._h, None if start is None else ctypes.c_void_p(start.cuda_event),
            None if stop is None else ctypes.c_void_p(stop.cuda_event)))

    def set_append_events(self, start: torch.cuda.Event | None,
                          stop: torch.cuda.Event | None) -> None:
        """Record these events around every KV append kernel launch of this stream."""
        _check(lib().frt_stream_set_append_events(
            self._h, None if start is None else ctypes.c_void_p(start.cuda_event),
            None if stop is None else ctypes.c_void_p(stop.cuda_event)))

    def check_guards(self) -> None:
        """Wait for the stream and compare the guard words around its KV cache."""
        _check(lib().frt_stream_check_guards(self._h))

    def save(self):
        """Snapshot of the persistent state: (k, v, counter), k and v device copies of
        the whole ring. Complete once sync() returns."""
        rows = self.window * self.n_q
        k = torch.empty((rows, self.heads, self.head_dim), dtype=torch.bfloat16, device="cuda")
        v = torch.empty_like(k)
        c = ctypes.c_longlong()
        _check(lib().frt_stream_save(self._h, _ptr(k), _ptr(v), ctypes.byref(c)))
        return k, v, c.value

    def restore(self, k: torch.Tensor, v: torch.Tensor, counter: int) -> None:
        """Continue from a snapshot taken by save() (of this or another stream of the same
        shape)."""
        rows = self.window * self.n_q
        _bf16_dev(k, (rows, self.heads, self.head_dim), "k")
        _bf16_dev(v, (rows, self.heads, self.head_dim), "v")
        _check(lib().frt_stream_restore(self._h, _ptr(k), _ptr(v), counter))

    def cache(self):
        """(k_cache, v_cache) device tensors viewing the stream's ring buffer
        [W * Nq, heads, head_dim] bf16 (read-only use)."""
        kp, vp = ctypes.c_void_p(), ctypes.c_void_p()
        rows = ctypes.c_longlong()
        _check(lib().frt_stream_cache(self._h, ctypes.byref(kp), ctypes.byref(vp),
                                      ctypes.byref(rows)))
        return (_view_bf16(kp.value, (rows.value, self.heads, self.head_dim)),
                _view_bf16(vp.value, (rows.value, self.heads, self.head_dim)))

    def _check_out(self, out):
        if out.dtype != self.out_dtype or not out.is_cuda or not out.is_contiguous() or \
                tuple(out.shape) != self.shape():
            raise ValueError("out must be a contiguous CUDA tensor of the stream's out dtype/shape")


def _view_bf16(ptr: int, shape) -> torch.Tensor:
    """Non-owning torch view of library-owned device memory."""
    n = 1
    for s in shape:
        n *= s

    class _Holder:
        __cuda_array_interface__ = {"shape": (n,), "typestr": "<u2", "data": (ptr, False),
                                    "version": 3, "strides": None}

    t = torch.as_tensor(_Holder(), device="cuda")
    return t.view(torch.bfloat16).view(*shape)


class ConvStream:
    """A streaming causal 3D convolution layer (its frame cache lives in the library)."""

    def __init__(self, cin: int, cout: int, kt: int, kh: int, kw: int, grid_h: int,
                 grid_w: int, frames_per_chunk: int, out_dtype: torch.dtype = torch.float32,
                 cuda_stream: torch.cuda.Stream | None = None):
        L = lib()
        self._h = L.frt_conv_create(cin, cout, kt, kh, kw, grid_h, grid_w, frames_per_chunk)
        if not self._h:
            raise FrtError(1, L.frt_last_error().decode())
        self.cin, self.cout, self.kt, self.kh, self.kw = cin, cout, kt, kh, kw
        self.grid_h, self.grid_w, self.frames = grid_h, grid_w, frames_per_chunk
        self.out_dtype = out_dtype
        self.torch_stream = cuda_stream or torch.cuda.current_stream()
        _check(L.frt_conv_configure(self._h, OUT_BF16 if out_dtype == torch.bfloat16 else OUT_F32,
                                    ctypes.c_void_p(self.torch_stream.cuda_stream)))

    def new_out(self) -> torch.Tensor:
        return torch.empty(self.frames, self.grid_h, self.grid_w, self.cout, dtype=self.out_dtype,
                           device="cuda")

    def step(self, x: torch.Tensor, w: torch.Tensor, bias: torch.Tensor, y: torch.Tensor) -> None:
        _bf16_dev(x, (self.frames, self.grid_h, self.grid_w, self.cin), "x")
        _bf16_dev(w, (self.kt * self.kh * self.kw, self.cout, self.cin), "w")
        if bias.dtype != torch.float32 or not bias.is_cuda or tuple(bias.shape) != (self.cout,):
            raise ValueError("bias must be a float32 CUDA tensor [Cout]")
        if y.dtype != self.out_dtype or not y.is_cuda or not y.is_contiguous() or \
                tuple(y.shape) != (self.frames, self.grid_h, self.grid_w, self.cout):
            raise ValueError("y must be a contiguous [F, H, W, Cout] CUDA tensor of the out dtype")
        _check(lib().frt_conv_step(self._h, _ptr(x), _ptr(w), _ptr(bias), _ptr(y)))

    def set_tile(self, bn: int = 0, pair: int = 0) -> None:
        """Force the kernel's output-channel tile and CTA pairing (bn = 0: automatic)."""
        _check(lib().frt_conv_set_tile(self._h, bn, pair))

    def set_split(self, mode: int = 0, units: int = 0) -> None:
        """Force the kernel's work split: 0 automatic, 1 whole tiles, 2 split tiles'
        halo steps over the units; units = 0 for every SM (or SM pair)."""
        _check(lib().frt_conv_set_split(self._h, mode, units))

    def cache(self) -> torch.Tensor:
        p = ctypes.c_void_p()
        _check(lib().frt_conv_cache(self._h, ctypes.byref(p)))
        return _view_bf16(p.value, (max(1, self.kt - 1), self.grid_h, self.grid_w, self.cin))

    def sync(self) -> None:
        _check(lib().frt_conv_sync(self._h))

    def reset(self) -> None:
        _check(lib().frt_conv_reset(self._h))

    def close(self) -> None:
        if getattr(self, "_h", None):
            lib().frt_conv_destroy(self._h)
            self._h = None

    def __del__(self):  # pragma: no cover - best effort
        try:
            self.close()
        except Exception:
            pass


def chunk_attention_batched(streams, qs, outs) -> None:
    n = len(streams)
    for s, q, o in zip(streams, qs, outs):
        _bf16_dev(q, s.shape(), "q")
        s._check_out(o)
    arr = ctypes.c_void_p * n
    _check(lib().frt_chunk_attention_batched(
        arr(*[s.handle for s in streams]), n, arr(*[q.data_ptr() for q in qs]),
        arr(*[o.data_ptr() for o in outs])))


class Steps:
    """Per-denoising-step caches: n_steps independent streams of one shape advanced by
    pipeline ticks (frt_steps_* in include/frt.h)."""

    def __init__(self, n_steps: int, heads: int, head_dim: int, grid_h: int, grid_w: int,
                 frames_per_chunk: int, window_chunks: int, split=None, theta: float = 10000.0,
                 out_dtype: torch.dtype = torch.float32):
        L = lib()
        self._g = L.frt_steps_create(n_steps, heads, head_dim, grid_h * grid_w,
                                     frames_per_chunk, window_chunks)
        if not self._g:
            raise FrtError(1, L.frt_last_error().decode())
        self.n_steps = n_steps
        self.n_q = frames_per_chunk * grid_h * grid_w
        self.heads, self.head_dim, self.out_dtype = heads, head_dim, out_dtype
        cfg = Config()
        _check(L.frt_config_default(L.frt_steps_stream(self._g, 0), ctypes.byref(cfg)))
        cfg.grid_h, cfg.grid_w = grid_h, grid_w
        if split is not None:
            cfg.rope_dt, cfg.rope_dh, cfg.rope_dw = (int(x) for x in split)
        cfg.theta = theta
        cfg.out_dtype = OUT_BF16 if out_dtype == torch.bfloat16 else OUT_F32
        cfg.cuda_stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
        _check(L.frt_steps_configure(self._g, ctypes.byref(cfg)))

    def shape(self):
        return (self.n_q, self.heads, self.head_dim)

    def counter(self, step: int) -> int:
        return lib().frt_stream_chunk_counter(lib().frt_steps_stream(self._g, step))

    def tick(self, active, q, k, v, out) -> None:
        """active: iterable of step indices; q/k/v/out: dicts or lists indexed by step."""
        arr = ctypes.c_void_p * self.n_steps
        mask = 0
        ptrs = {n: [None] * self.n_steps for n in ("q", "k", "v", "o")}
        for i in active:
            mask |= 1 << i
            for n, t in (("q", q[i]), ("k", k[i]), ("v", v[i])):
                _bf16_dev(t, self.shape(), n)
                ptrs[n][i] = t.data_ptr()
            ptrs["o"][i] = out[i].data_ptr()
        _check(lib().frt_steps_tick(self._g, mask, arr(*ptrs["q"]), arr(*ptrs["k"]),
                                    arr(*ptrs["v"]), arr(*ptrs["o"])))

    def sync(self) -> None:
        for i in range(self.n_steps):
            _check(lib().frt_stream_sync(lib().frt_steps_stream(self._g, i)))

    def close(self) -> None:
        if getattr(self, "_g", None):
            lib().frt_steps_destroy(self._g)
            self._g = None

    def __del__(self):  # pragma: no cover - best effort
        try:
            self.close()
        except Exception:
            pass


def selftest_gemm_force_bn(bn: int) -> None:
    """Force the projection kernel's tile width (128, 192 or 256; 0 = automatic)."""
    if lib().frt_selftest_gemm_force_bn(bn) != 0:
        raise ValueError("bn must be 0, 128, 192 or 256")


def selftest_conv_part_mode(mode: int) -> None:
    """How split convolution tiles gather their parts (0 as built, 1 no watch, 2 no
    watch and no wait: the first part writes itself and arrives)."""
    if lib().frt_selftest_conv_part_mode(mode) != 0:
        raise ValueError("mode must be 0, 1 or 2")


def gemm_plan(M: int, N: int, qkv: bool = False, d: int = 0) -> tuple[int, int]:
    """(output columns per tile, CTAs per tile) the projection kernel uses for C [M, N]."""
    bn, ctas = ctypes.c_int(), ctypes.c_int()
    _check(lib().frt_gemm_plan(M, N, 1 if qkv else 0, d, ctypes.byref(bn), ctypes.byref(ctas)))
    return bn.value, ctas.value


def attention_plan(n_q, n_kv, heads: int, sms: int = 0) -> tuple[int, int]:
    """(n_full, n_split) of one attention launch over streams with n_q[i] queries and
    n_kv[i] valid keys (launch order): query groups [0, n_full) run whole, later ones are
    cut into n_split KV parts."""
    n = len(n_q)
    a = (ctypes.c_int * n)(*n_q)
    b = (ctypes.c_longlong * n)(*n_kv)
    nf, ns = ctypes.c_int(), ctypes.c_int()
    _check(lib().frt_attention_plan(n, a, b, heads, sms, ctypes.byref(nf), ctypes.byref(ns)))
    return nf.value, ns.value


def conv_plan(cin: int, cout: int, kt: int, kh: int, kw: int, grid_h: int, grid_w: int,
              frames: int, sms: int, out_dtype=torch.float32, bn: int = 0, pair: int = 0,
              split_mode: int = 0, units: int = 0) -> dict:
    """The launch plan of frt_conv_step for these sizes on `sms` SMs (host-only)."""
    plan = (ctypes.c_int * 6)()
    _check(lib().frt_conv_plan(cin, cout, kt, kh, kw, grid_h, grid_w, frames,
                               OUT_BF16 if out_dtype == torch.bfloat16 else OUT_F32, sms, bn,
                               pair, split_mode, units, plan))
    return dict(bn=plan[0], pair=plan[1], units=plan[2], split=plan[3], n_tiles=plan[4],
                nhalo=plan[5])


def gemm_bf16(a: torch.Tensor, b: torch.Tensor, c: torch.Tensor,
              status: torch.Tensor | None = None) -> None:
    """c[:M, :N] = a @ b.T on the tensor cores (a [M, K], b [N, K] bf16; c fp32 or bf16,
    row stride c.stride(0)); enqueued on torch's current CUDA stream."""
    for t, n in ((a, "a"), (b, "b")):
        if t.dtype != torch.bfloat16 or not t.is_cuda or not t.is_contiguous() or t.dim() != 2:
            raise ValueError(f"{n} must be a contiguous 2D bf16 CUDA tensor")
    M, K = a.shape
    N = b.shape[0]
    if b.shape[1] != K:
        raise ValueError("a and b disagree on K")
    if c.dim() != 2 or c.stride(1) != 1 or not c.is_cuda or c.shape[0] < M or c.shape[1] < N:
        raise ValueError("c must be a row-major CUDA matrix of at least [M, N]")
    if c.dtype == torch.float32:
        cd = OUT_F32
    elif c.dtype == torch.bfloat16:
        cd = OUT_BF16
    else:
        raise ValueError("c must be float32 or bfloat16")
    _check(lib().frt_gemm_bf16(_ptr(a), _ptr(b), _ptr(c), M, N, K, c.stride(0), cd,
                               _ptr(status),
                               ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)))


def selftest_umma_tile(a: torch.Tensor, b: torch.Tensor, b_mn_major: bool, lbo: int = 16384,
                       sbo: int = 1024, a_from_tmem: bool = False) -> torch.Tensor:
    c = torch.empty(128, 128, dtype=torch.float32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    rc = lib().frt_selftest_umma_tile(_ptr(a), _ptr(b), _ptr(c), int(b_mn_major), lbo, sbo,
                                      int(a_from_tmem), _ptr(status),
                                      ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    if rc != 0:
        raise FrtError(4, f"selftest launch failed ({rc})")
    torch.cuda.synchronize()
    if int(status.item()) != 0:
        raise FrtError(6, "selftest tile timed out")
    return c


def selftest_umma_pair(a: torch.Tensor, b: torch.Tensor, pv: bool = False):
    """(C [256,128] fp32, TMEM addresses the two CTAs got) for C = A B^T on a CTA pair, or
    with pv=True C = A B with A staged in TMEM and B read MN-major (the P.V form)."""
    c = torch.empty(256, 128, dtype=torch.float32, device="cuda")
    taddrs = torch.zeros(2, dtype=torch.int32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    fn = lib().frt_selftest_umma_pair_pv if pv else lib().frt_selftest_umma_pair
    rc = fn(_ptr(a), _ptr(b), _ptr(c), _ptr(taddrs), _ptr(status),
            ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    if rc != 0:
        raise FrtError(4, f"pair selftest launch failed ({rc})")
    torch.cuda.synchronize()
    if int(status.item()) != 0:
        raise FrtError(6, "pair selftest timed out")
    return c, taddrs.cpu().tolist()


def selftest_wait_timeout(stream: Stream, limit_ns: int) -> None:
    _check(lib().frt_selftest_wait_timeout(
        stream.handle, limit_ns, ctypes.c_void_p(stream.torch_stream.cuda_stream)))
