"""CPU oracle for the spike-gated INT8 projection (Section 2.3, Eq. sparse).

TEST INFRASTRUCTURE ONLY.  Only the test suite, ``__graft_entry__.smoke()``
and the CPU-baseline leg of ``bench.py`` may import this package.  The CUDA
library never calls it, and the two share no code: this wrapper compiles
``spike_oracle.c`` with the host C compiler and calls it through ctypes.

Functions mirror ``spike_oracle.h``:

* :func:`active_set` -- ``A = {k : x_k = 1}``, ascending (Section 2.2).
* :func:`project` -- ``acc_m = sum_{k in A} Q[k*ldq + m]`` in int64 narrowed
  to INT32, ``y_m = s_m * float32(acc_m)`` (Eq. sparse and the sentence after
  it), for T spike rows.
* :func:`project_entries` -- the same at selected (row, channel) pairs.
* :func:`lif` -- one leaky integrate-and-fire step producing spike rows in
  the ``"bits"`` format (a stated reading: the paper names LIF only).
* :func:`dense` -- the continuous-input projection over row-major INT8
  weights, ``y_m = s_m * sum_k Q[m*ldq + k] * x_k`` evaluated in double, with
  ``sum_k |Q_mk x_k|`` for error bounds (Section 2.3, the sentence on
  continuous inputs; Section 2.2 for the row-major layout).
* :func:`head` -- the vocabulary head with INT8 activations, the top-two
  gap gate and FP32-activation recomputation of the top candidates
  (Section 5, trace configuration; Appendix D; the activation quantiser is a
  stated reading).

Spike formats: ``"bits"`` = uint32 words, column k is bit k%32 of word k//32
(LSB first, tail bits ignored); ``"u8"`` = one byte per column, nonzero fires.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from pathlib import Path

import numpy as np

_HERE = Path(__file__).resolve().parent
_SRC = _HERE / "spike_oracle.c"
_HDR = _HERE / "spike_oracle.h"
_OUT_DIR = _HERE / "_build"
_LIB = _OUT_DIR / "libspike_oracle.so"

FMT_BITS = 0
FMT_U8 = 1
_FMTS = {"bits": FMT_BITS, "u8": FMT_U8}

# -O2 with FP contraction off: the only float operation is one multiply per
# output, but the flag keeps any compiler from fusing it with anything.
CFLAGS = ["-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math",
          "-fPIC", "-shared", "-Wall", "-Wextra"]


def build(force: bool = False, cc: str | None = None) -> Path:
    """Compile the oracle into ``oracle/_build/libspike_oracle.so``."""
    _OUT_DIR.mkdir(exist_ok=True)
    newest = max(_SRC.stat().st_mtime, _HDR.stat().st_mtime)
    if not force and _LIB.exists() and _LIB.stat().st_mtime >= newest:
        return _LIB
    cc = cc or os.environ.get("CC", "gcc")
    tmp = _LIB.with_suffix(f".so.tmp{os.getpid()}")
    subprocess.run([cc, *CFLAGS, "-o", str(tmp), str(_SRC)], check=True)
    os.replace(tmp, _LIB)
    return _LIB


def compile_source(src_text: str, out: Path, cc: str | None = None) -> Path:
    """Compile an oracle source text (used by tests that plant a mistake in
    a copy of the oracle and check that the pins catch it)."""
    out = Path(out)
    c_file = out.with_suffix(".c")
    c_file.write_text(src_text)
    hdr = out.parent / "spike_oracle.h"
    hdr.write_text(_HDR.read_text())
    cc = cc or os.environ.get("CC", "gcc")
    subprocess.run([cc, *CFLAGS, "-o", str(out), str(c_file)], check=True)
    return out


class Oracle:
    """ctypes handle on one compiled oracle library."""

    def __init__(self, path: Path | str | None = None):
        self.path = Path(path) if path else build()
        lib = ctypes.CDLL(str(self.path))
        p, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
        lib.sp_oracle_active_set.argtypes = [p, ctypes.c_int, i32, p, p]
        lib.sp_oracle_active_set.restype = ctypes.c_int
        lib.sp_oracle_project.argtypes = [p, i64, p, i32, i32, p, ctypes.c_int,
                                          i64, i32, p, p]
        lib.sp_oracle_project.restype = ctypes.c_int
        lib.sp_oracle_project_entries.argtypes = [p, i64, p, i32, i32, p,
                                                  ctypes.c_int, i64, i32, i64,
                                                  p, p, p, p]
        lib.sp_oracle_project_entries.restype = ctypes.c_int
        lib.sp_oracle_dense.argtypes = [p, i64, p, i32, i32, p, i64, i32, p, p]
        lib.sp_oracle_dense.restype = ctypes.c_int
        lib.sp_oracle_lif.argtypes = [p, p, i32, i32, i64, ctypes.c_float, ctypes.c_float, p, i64]
        lib.sp_oracle_lif.restype = ctypes.c_int
        lib.sp_oracle_head.argtypes = [p, i64, p, i32, i32, p, i64, i32, ctypes.c_float, i32,
                                       p, p, p, p, p, p, p, p, p]
        lib.sp_oracle_head.restype = ctypes.c_int
        self.lib = lib

    # -- helpers -----------------------------------------------------------
    @staticmethod
    def _spikes(spikes: np.ndarray, fmt: str, K: int):
        if fmt not in _FMTS:
            raise ValueError(f"unknown spike format {fmt!r}")
        if fmt == "bits":
            spikes = np.ascontiguousarray(spikes, dtype=np.uint32)
            if spikes.ndim == 1:
                spikes = spikes[None, :]
            if spikes.shape[1] < (K + 31) // 32:
                raise ValueError("bit rows shorter than ceil(K/32) words")
        else:
            spikes = np.ascontiguousarray(spikes, dtype=np.uint8)
            if spikes.ndim == 1:
                spikes = spikes[None, :]
            if spikes.shape[1] < K:
                raise ValueError("u8 rows shorter than K")
        return spikes, _FMTS[fmt], spikes.shape[1]

    @staticmethod
    def _weights(Q: np.ndarray, scale: np.ndarray | None, N: int, K: int,
                 ldq: int | None):
        Q = np.ascontiguousarray(Q, dtype=np.int8).reshape(-1)
        ldq = N if ldq is None else ldq
        if ldq < N or Q.size < ldq * (K - 1) + N:
            raise ValueError("Q too small for N, K, ldq")
        if scale is not None:
            scale = np.ascontiguousarray(scale, dtype=np.float32).reshape(-1)
            if scale.size < N:
                raise ValueError("scale shorter than N")
        return Q, scale, ldq

    # -- API -----------------------------------------------------------------
    def active_set(self, spikes: np.ndarray, fmt: str, K: int) -> np.ndarray:
        sp, f, _ = self._spikes(spikes, fmt, K)
        idx = np.zeros(max(K, 1), dtype=np.int32)
        cnt = ctypes.c_int32(0)
        rc = self.lib.sp_oracle_active_set(sp.ctypes.data, f, K,
                                           idx.ctypes.data,
                                           ctypes.addressof(cnt))
        if rc:
            raise RuntimeError(f"sp_oracle_active_set failed: {rc}")
        return idx[: cnt.value].copy()

    def project(self, Q: np.ndarray, scale: np.ndarray, N: int, K: int,
                spikes: np.ndarray, fmt: str, ldq: int | None = None):
        """Eq. (sparse) for every row of ``spikes``; returns (acc, y) shaped
        [T, N] (int32, float32)."""
        Q, scale, ldq = self._weights(Q, scale, N, K, ldq)
        sp, f, ld = self._spikes(spikes, fmt, K)
        T = sp.shape[0]
        acc = np.zeros((T, N), dtype=np.int32)
        y = np.zeros((T, N), dtype=np.float32)
        rc = self.lib.sp_oracle_project(Q.ctypes.data, ldq, scale.ctypes.data,
                                        N, K, sp.ctypes.data, f, ld, T,
                                        acc.ctypes.data, y.ctypes.data)
        if rc:
            raise RuntimeError(f"sp_oracle_project failed: {rc}")
        return acc, y

    def project_entries(self, Q: np.ndarray, scale: np.ndarray, N: int, K: int,
                        spikes: np.ndarray, fmt: str, t_idx, m_idx,
                        ldq: int | None = None):
        """Eq. (sparse) at (t_idx[e], m_idx[e]); returns (acc, y) of length
        len(t_idx)."""
        Q, scale, ldq = self._weights(Q, scale, N, K, ldq)
        sp, f, ld = self._spikes(spikes, fmt, K)
        t_idx = np.ascontiguousarray(t_idx, dtype=np.int32)
        m_idx = np.ascontiguousarray(m_idx, dtype=np.int32)
        if t_idx.shape != m_idx.shape:
            raise ValueError("t_idx and m_idx differ in shape")
        n = t_idx.size
        acc = np.zeros(n, dtype=np.int32)
        y = np.zeros(n, dtype=np.float32)
        rc = self.lib.sp_oracle_project_entries(
            Q.ctypes.data, ldq, scale.ctypes.data, N, K, sp.ctypes.data, f, ld,
            sp.shape[0], n, t_idx.ctypes.data, m_idx.ctypes.data,
            acc.ctypes.data, y.ctypes.data)
        if rc:
            raise RuntimeError(f"sp_oracle_project_entries failed: {rc}")
        return acc, y


    def dense(self, Q: np.ndarray, scale: np.ndarray, N: int, K: int,
              x: np.ndarray, ldq: int | None = None):
        """Continuous-input projection of every row of ``x`` (float32 [T, >=K])
        through row-major ``Q`` ([N, ldq] int8); returns (y, abs_dot), both
        float64 [T, N]."""
        ldq = K if ldq is None else ldq
        Q = np.ascontiguousarray(Q, dtype=np.int8).reshape(-1)
        if ldq < K or Q.size < ldq * (N - 1) + K:
            raise ValueError("Q too small for N, K, ldq")
        scale = np.ascontiguousarray(scale, dtype=np.float32).reshape(-1)
        if scale.size < N:
            raise ValueError("scale shorter than N")
        x = np.ascontiguousarray(x, dtype=np.float32)
        if x.ndim == 1:
            x = x[None, :]
        if x.shape[1] < K:
            raise ValueError("x rows shorter than K")
        T = x.shape[0]
        y = np.zeros((T, N), dtype=np.float64)
        mag = np.zeros((T, N), dtype=np.float64)
        rc = self.lib.sp_oracle_dense(Q.ctypes.data, ldq, scale.ctypes.data, N, K,
                                      x.ctypes.data, x.shape[1], T, y.ctypes.data,
                                      mag.ctypes.data)
        if rc:
            raise RuntimeError(f"sp_oracle_dense failed: {rc}")
        return y, mag


    def lif(self, v: np.ndarray, I: np.ndarray, K: int, beta: float, theta: float):
        """One LIF step of every row of ``v`` / ``I`` (float32 [T, >=K]);
        returns (v_new float32 [T, ld], bits uint32 [T, ceil(K/32)])."""
        v = np.array(v, dtype=np.float32, copy=True, ndmin=2, order="C")
        I = np.ascontiguousarray(I, dtype=np.float32)
        if I.ndim == 1:
            I = I[None, :]
        if v.shape != I.shape or v.shape[1] < K:
            raise ValueError("v and I must have the same shape, rows >= K")
        T, ld = v.shape
        words = (K + 31) // 32
        bits = np.full((T, max(words, 1)), 0xA5A5A5A5, dtype=np.uint32)
        rc = self.lib.sp_oracle_lif(v.ctypes.data, I.ctypes.data, K, T, ld, beta, theta,
                                    bits.ctypes.data, bits.shape[1])
        if rc:
            raise RuntimeError(f"sp_oracle_lif failed: {rc}")
        return v, bits[:, :words]


    def head(self, Q: np.ndarray, scale: np.ndarray, V: int, K: int, h: np.ndarray,
             tau: float, k_sel: int, ldq: int | None = None) -> dict:
        """Vocabulary head for every row of ``h`` (float32 [B, >=K]) through
        row-major ``Q`` ([V, ldq] int8).  Returns a dict of numpy arrays:
        codes int8 [B, K], s_x float32 [B], z float32 [B, V], gap float32 [B],
        verified int32 [B], cand int32 [B, k_sel], r / r_abs float64
        [B, k_sel], token int32 [B]."""
        ldq = K if ldq is None else ldq
        Q = np.ascontiguousarray(Q, dtype=np.int8).reshape(-1)
        if ldq < K or Q.size < ldq * (V - 1) + K:
            raise ValueError("Q too small for V, K, ldq")
        scale = np.ascontiguousarray(scale, dtype=np.float32).reshape(-1)
        if scale.size < V:
            raise ValueError("scale shorter than V")
        h = np.ascontiguousarray(h, dtype=np.float32)
        if h.ndim == 1:
            h = h[None, :]
        if h.shape[1] < K:
            raise ValueError("h rows shorter than K")
        B = h.shape[0]
        out = {"codes": np.zeros((B, K), np.int8), "s_x": np.zeros(B, np.float32),
               "z": np.zeros((B, V), np.float32), "gap": np.zeros(B, np.float32),
               "verified": np.zeros(B, np.int32), "cand": np.zeros((B, k_sel), np.int32),
               "r": np.zeros((B, k_sel), np.float64), "r_abs": np.zeros((B, k_sel), np.float64),
               "token": np.zeros(B, np.int32)}
        o = out
        rc = self.lib.sp_oracle_head(Q.ctypes.data, ldq, scale.ctypes.data, V, K, h.ctypes.data,
                                     h.shape[1], B, tau, k_sel, o["codes"].ctypes.data,
                                     o["s_x"].ctypes.data, o["z"].ctypes.data,
                                     o["gap"].ctypes.data, o["verified"].ctypes.data,
                                     o["cand"].ctypes.data, o["r"].ctypes.data,
                                     o["r_abs"].ctypes.data, o["token"].ctypes.data)
        if rc:
            raise RuntimeError(f"sp_oracle_head failed: {rc}")
        return out


_DEFAULT: Oracle | None = None


def default() -> Oracle:
    """The oracle built from ``spike_oracle.c`` (compiled on first use)."""
    global _DEFAULT
    if _DEFAULT is None:
        _DEFAULT = Oracle()
    return _DEFAULT


def active_set(spikes, fmt, K):
    return default().active_set(spikes, fmt, K)


def project(Q, scale, N, K, spikes, fmt, ldq=None):
    return default().project(Q, scale, N, K, spikes, fmt, ldq)


def project_entries(Q, scale, N, K, spikes, fmt, t_idx, m_idx, ldq=None):
    return default().project_entries(Q, scale, N, K, spikes, fmt, t_idx,
                                     m_idx, ldq)


def dense(Q, scale, N, K, x, ldq=None):
    return default().dense(Q, scale, N, K, x, ldq)


def lif(v, I, K, beta, theta):
    return default().lif(v, I, K, beta, theta)


def head(Q, scale, V, K, h, tau, k_sel, ldq=None):
    return default().head(Q, scale, V, K, h, tau, k_sel, ldq)
