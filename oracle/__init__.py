"""fp64 CPU oracle for softmax attention forward (ctypes wrapper of oracle.c).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
bench's ``cpu_baseline`` / ``--impl reference`` legs are the only callers.
The product path (``paper_2609_18077_gb300``) never imports this package,
and this package imports nothing from it.

What the oracle computes is the plain softmax-attention definition (vidax
paper, Sec. 2 "3D RoPE, 3D VAEs, and flash attention": flash attention is
an exact re-ordering of it), with padded text keys excluded per sample
(appendix Table 4, segment-id masking of invalid key blocks), either as a
valid key count per sample or as segment ids per token.  See the
header of ``oracle.c`` for the formulas.

Inputs are bf16 bit patterns as ``numpy.uint16`` arrays ``[B, H, S, D]``;
outputs are ``float64``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
SOURCE = os.path.join(_HERE, "oracle.c")
LIBRARY = os.path.join(_HERE, "liboracle.so")


def build(source: str = SOURCE, output: str = LIBRARY, extra_flags=()) -> str:
    """Compile ``oracle.c`` with gcc (fp64, OpenMP, no fast-math)."""
    cmd = ["gcc", "-O2", "-fopenmp", "-shared", "-fPIC", "-std=c99",
           *extra_flags, "-o", output, source, "-lm"]
    subprocess.run(cmd, check=True, capture_output=True, text=True)
    return output


class Oracle:
    """Handle on one compiled oracle library (the real one, or a test mutant)."""

    def __init__(self, path: str = LIBRARY):
        if not os.path.exists(path):
            raise FileNotFoundError(f"oracle library {path} is not built; call oracle.build()")
        self.path = path
        lib = ctypes.CDLL(path)
        lib.oracle_attn_fwd.restype = ctypes.c_int
        lib.oracle_attn_fwd.argtypes = [
            ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
            ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
            ctypes.c_double, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int,
            ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]
        lib.oracle_attn_fwd_seg.restype = ctypes.c_int
        lib.oracle_attn_fwd_seg.argtypes = [
            ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
            ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
            ctypes.c_double, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int,
            ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]
        lib.oracle_attn_fwd_win3d.restype = ctypes.c_int
        lib.oracle_attn_fwd_win3d.argtypes = [
            ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
            ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_double,
            ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
            ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]
        lib.oracle_rope3d.restype = ctypes.c_int
        lib.oracle_rope3d.argtypes = [
            ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
            ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
            ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_double, ctypes.c_int, ctypes.c_void_p]
        lib.oracle_set_threads.restype = ctypes.c_int
        lib.oracle_set_threads.argtypes = [ctypes.c_int]
        self._lib = lib

    def set_threads(self, n: int = 0) -> int:
        """Set the OpenMP thread count (n <= 0 keeps it); returns the count in use."""
        return int(self._lib.oracle_set_threads(int(n)))

    def attn_fwd(self, q, k, v, scale, kv_lens=None, rows=None, probs=False, q_seg=None, kv_seg=None):
        """Attention forward in fp64.

        q: uint16 [B,H,Sq,D]; k, v: uint16 [B,H,Skv,D] (bf16 bits).
        kv_lens: None or int [B] (valid keys per sample, clamped to [0, Skv]).
        rows: None (all query rows) or int [B*H, n] query indices per (b, h).
        q_seg, kv_seg: None, or int [B,Sq] and int [B,Skv] segment ids (given
        together, without kv_lens): a query attends the keys of its segment.
        Returns (o [B,H,n,D] f64, lse [B,H,n] f64[, probs [B,H,n,Skv] f64]).
        """
        q = _bits(q)
        k = _bits(k)
        v = _bits(v)
        B, H, Sq, D = q.shape
        Skv = k.shape[2]
        if k.shape != (B, H, Skv, D) or v.shape != (B, H, Skv, D):
            raise ValueError("k and v must be [B,H,Skv,D] matching q")
        lens = None
        if kv_lens is not None:
            lens = np.ascontiguousarray(np.asarray(kv_lens, dtype=np.int32))
            if lens.shape != (B,):
                raise ValueError("kv_lens must have shape [B]")
        if rows is None:
            n = Sq
            rows_arr = None
        else:
            rows_arr = np.ascontiguousarray(np.asarray(rows, dtype=np.int32))
            if rows_arr.ndim != 2 or rows_arr.shape[0] != B * H:
                raise ValueError("rows must have shape [B*H, n]")
            n = rows_arr.shape[1]
        if (q_seg is None) != (kv_seg is None):
            raise ValueError("q_seg and kv_seg go together")
        if q_seg is not None:
            if lens is not None:
                raise ValueError("segment ids and kv_lens are exclusive")
            qs = np.ascontiguousarray(np.asarray(q_seg, dtype=np.int32))
            ks = np.ascontiguousarray(np.asarray(kv_seg, dtype=np.int32))
            if qs.shape != (B, Sq) or ks.shape != (B, Skv):
                raise ValueError("q_seg must be [B,Sq] and kv_seg [B,Skv]")
        o = np.empty((B, H, n, D), dtype=np.float64)
        lse = np.empty((B, H, n), dtype=np.float64)
        pr = np.empty((B, H, n, Skv), dtype=np.float64) if probs else None
        if q_seg is None:
            rc = self._lib.oracle_attn_fwd(
                _ptr(q), _ptr(k), _ptr(v), B, H, Sq, Skv, D, float(scale),
                _ptr(lens), _ptr(rows_arr), n, _ptr(o), _ptr(lse), _ptr(pr))
        else:
            rc = self._lib.oracle_attn_fwd_seg(
                _ptr(q), _ptr(k), _ptr(v), B, H, Sq, Skv, D, float(scale),
                _ptr(qs), _ptr(ks), _ptr(rows_arr), n, _ptr(o), _ptr(lse), _ptr(pr))
        if rc != 0:
            raise RuntimeError("oracle attention rejected its arguments")
        return (o, lse, pr) if probs else (o, lse)


    def attn_fwd_win3d(self, q, k, v, scale, grid, window, neighbourhood=True, rows=None, probs=False):
        """Windowed 3D attention in fp64 (see oracle.c).

        q, k, v: uint16 [B,H,S,D] with S = F*Hp*Wp tokens of the grid (F, Hp, Wp)
        in raster order; window = (kt, kh, kw), odd sizes.
        Returns (o, lse[, probs]) like attn_fwd.
        """
        q, k, v = _bits(q), _bits(k), _bits(v)
        B, H, S, D = q.shape
        F, Hp, Wp = (int(x) for x in grid)
        if S != F * Hp * Wp or k.shape != q.shape or v.shape != q.shape:
            raise ValueError("q, k, v must be [B,H,F*Hp*Wp,D] alike")
        if rows is None:
            n, rows_arr = S, None
        else:
            rows_arr = np.ascontiguousarray(np.asarray(rows, dtype=np.int32))
            if rows_arr.ndim != 2 or rows_arr.shape[0] != B * H:
                raise ValueError("rows must have shape [B*H, n]")
            n = rows_arr.shape[1]
        o = np.empty((B, H, n, D), dtype=np.float64)
        lse = np.empty((B, H, n), dtype=np.float64)
        pr = np.empty((B, H, n, S), dtype=np.float64) if probs else None
        rc = self._lib.oracle_attn_fwd_win3d(_ptr(q), _ptr(k), _ptr(v), B, H, F, Hp, Wp, D, float(scale),
                                             int(window[0]), int(window[1]), int(window[2]), int(bool(neighbourhood)),
                                             _ptr(rows_arr), n, _ptr(o), _ptr(lse), _ptr(pr))
        if rc != 0:
            raise RuntimeError("oracle_attn_fwd_win3d rejected its arguments")
        return (o, lse, pr) if probs else (o, lse)

    def rope3d(self, x, grid, s0, dims, theta, interleaved=True):
        """3D rotary embedding in fp64 (see oracle.c).

        x: uint16 [B,H,S,D] bf16 bits; grid = (F, Hp, Wp); tokens [s0, s0+F*Hp*Wp)
        are the video grid; dims = (d_t, d_h, d_w).  Returns float64 [B,H,S,D].
        """
        x = _bits(x)
        B, H, S, D = x.shape
        F, Hp, Wp = grid
        y = np.empty((B, H, S, D), dtype=np.float64)
        rc = self._lib.oracle_rope3d(_ptr(x), B, H, S, D, int(F), int(Hp), int(Wp), int(s0),
                                     int(dims[0]), int(dims[1]), int(dims[2]), float(theta), int(bool(interleaved)),
                                     _ptr(y))
        if rc != 0:
            raise RuntimeError("oracle_rope3d rejected its arguments")
        return y


def _bits(a) -> np.ndarray:
    a = np.asarray(a)
    if a.dtype != np.uint16 or a.ndim != 4:
        raise TypeError("oracle inputs are uint16 bf16 bit patterns of rank 4")
    return np.ascontiguousarray(a)


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


_default = None


def default() -> Oracle:
    """The oracle built from ``oracle.c`` (compiled on first use if missing)."""
    global _default
    if _default is None:
        if not os.path.exists(LIBRARY) or os.path.getmtime(LIBRARY) < os.path.getmtime(SOURCE):
            build()
        _default = Oracle(LIBRARY)
    return _default


def attn_fwd_win3d(q, k, v, scale, grid, window, neighbourhood=True, rows=None, probs=False):
    """Module-level shortcut for ``default().attn_fwd_win3d``."""
    return default().attn_fwd_win3d(q, k, v, scale, grid, window, neighbourhood, rows, probs)


def rope3d(x, grid, s0, dims, theta, interleaved=True):
    """Module-level shortcut for ``default().rope3d``."""
    return default().rope3d(x, grid, s0, dims, theta, interleaved)


def attn_fwd(q, k, v, scale, kv_lens=None, rows=None, probs=False, q_seg=None, kv_seg=None):
    """Module-level shortcut for ``default().attn_fwd``."""
    return default().attn_fwd(q, k, v, scale, kv_lens=kv_lens, rows=rows, probs=probs, q_seg=q_seg,
                              kv_seg=kv_seg)
