"""ctypes binding of libspikeproj.so (``include/spike_proj.h``).

Argument marshalling only: every step of the projection runs in the CUDA
library.  Functions keep the C names; device buffers are passed as torch CUDA
tensors (or raw integer device addresses), streams default to torch's current
stream.  A missing library is an error, never a fallback.
"""
from __future__ import annotations

import ctypes
from pathlib import Path

LIB_PATH = Path(__file__).resolve().parent / "_build" / "libspikeproj.so"

# sp_status
SP_OK, SP_EINVAL, SP_EALIGN, SP_EDEVICE, SP_ECUDA, SP_ENOMEM, SP_ERANGE, \
    SP_EKERNEL, SP_EUNSUPPORTED, SP_ESCRATCH = range(10)
# sp_fmt
SP_SPIKES_BITS32, SP_SPIKES_U8, SP_SPIKES_BOOL8 = 0, 1, 2
# sp_kernel
SP_AUTO, SP_GATHER, SP_UNION, SP_GEMM = 0, 1, 2, 3
# sp_fault (tests of the error path only)
SP_FAULT_NONE, SP_FAULT_ABORT, SP_FAULT_STALL = 0, 1, 2
SP_PLAN_GEMM = 0x1
SPIKE_PROJ_MAX_K = 131072
SPIKE_PROJ_MAX_GROUP = 64
SPIKE_PROJ_NOALLOC_MAX_N = 32768
SPIKE_PROJ_DENSE_MAX_B = 4
SPIKE_PROJ_DENSE_MAX_GROUP = 128

FMTS = {"bits": SP_SPIKES_BITS32, "u8": SP_SPIKES_U8, "bool8": SP_SPIKES_BOOL8}
KERNELS = {"auto": SP_AUTO, "gather": SP_GATHER, "union": SP_UNION, "gemm": SP_GEMM}
KERNEL_NAMES = {v: k for k, v in KERNELS.items()}

# every entry point of the C ABI with its ctypes signature
_P, _I32, _I64, _U32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32
_SIGNATURES = {
    "spike_proj_plan": ([_P, _P, _I64, _P, _I32, _I32, _I32, _U32, _P], ctypes.c_int),
    "spike_proj_plan_destroy": ([_P], ctypes.c_int),
    "spike_proj_decode": ([_P, _P, ctypes.c_int, _P, _P, _P], ctypes.c_int),
    "spike_proj_batched": ([_P, _P, ctypes.c_int, _I32, _I64, _P, _P, ctypes.c_int, _P],
                           ctypes.c_int),
    "spike_proj_prefill": ([_P, _P, _I32, _I64, _P, _P, ctypes.c_int, _P], ctypes.c_int),
    "spike_proj_last_dispatch": ([_P, _P, _P], ctypes.c_int),
    "spike_proj_plan_status": ([_P, _P], ctypes.c_int),
    "spike_proj_group_create": ([_P, _P, _I32, _P], ctypes.c_int),
    "spike_proj_group_destroy": ([_P], ctypes.c_int),
    "spike_proj_group_decode": ([_P, _P, ctypes.c_int, _I64, _P, _P, _I64, _P], ctypes.c_int),
    "spike_proj_group_decode_host": ([_P, _P, ctypes.c_int, _I64, _P, _P, _I64, _P],
                                     ctypes.c_int),
    "spike_proj_group_decode_lif": ([_P, _P, _P, _P, _I64, ctypes.c_float, ctypes.c_float, _P,
                                     _I64, _P, _P, _I64, _P], ctypes.c_int),
    "spike_proj_group_status": ([_P, _P], ctypes.c_int),
    "spike_proj_group_prefill": ([_P, _P, ctypes.c_int, _I32, _I64, _P, _P, _P], ctypes.c_int),
    "spike_proj_decode_noalloc": ([_P, _I64, _P, _I32, _I32, _P, ctypes.c_int, _P, _P, _P],
                                  ctypes.c_int),
    "spike_proj_dense": ([_P, _I32, _I32, _P], ctypes.c_int),
    "spike_proj_lif": ([_P, _P, _I32, _I32, _I64, ctypes.c_float, ctypes.c_float, _P, _I64, _P],
                       ctypes.c_int),
    "spike_proj_head_create": ([_P, _P, _I64, _P, _I32, _I32, _P], ctypes.c_int),
    "spike_proj_head_destroy": ([_P], ctypes.c_int),
    "spike_proj_head": ([_P, _P, _I64, _I32, ctypes.c_float, _I32, _P, _P, _P, _P, _P, _P, _I64,
                         _P], ctypes.c_int),
    "spike_proj_probe_gather": ([_P, _P, _I32, _I32, _P, _P], ctypes.c_int),
    "spike_proj_plan_inject_fault": ([_P, _I32], ctypes.c_int),
    "spike_proj_group_inject_fault": ([_P, _I32], ctypes.c_int),
    "spike_proj_strerror": ([ctypes.c_int], ctypes.c_char_p),
    "spike_proj_last_cuda_error": ([], ctypes.c_int),
    "spike_proj_abi_version": ([], ctypes.c_int),
}

_lib = None


class SpikeProjError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        msg = lib().spike_proj_strerror(status).decode()
        if status == SP_ECUDA:
            msg += f" (cudaError {lib().spike_proj_last_cuda_error()})"
        super().__init__(f"{where}: {msg} [status {status}]")


def lib():
    """The loaded library (opened on first use).  Raises if it is not built."""
    global _lib
    if _lib is None:
        if not LIB_PATH.exists():
            raise RuntimeError(
                f"{LIB_PATH} is missing: build the CUDA library first "
                "(python -c 'import __graft_entry__ as g; g.build()')")
        L = ctypes.CDLL(str(LIB_PATH))
        for name, (args, res) in _SIGNATURES.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = res
        _lib = L
    return _lib


def _addr(x):
    """Device (or host) address of a tensor / numpy array / int / None."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if hasattr(x, "ctypes"):
        return x.ctypes.data
    raise TypeError(f"cannot take the address of {type(x)!r}")


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(status: int, where: str):
    if status != SP_OK:
        raise SpikeProjError(status, where)


def _fmt(fmt):
    return FMTS[fmt] if isinstance(fmt, str) else int(fmt)


def _kernel(k):
    return KERNELS[k] if isinstance(k, str) else int(k)


# ---------------------------------------------------------------------------
# thin wrappers, same names as the C ABI
# ---------------------------------------------------------------------------
def spike_proj_plan(W, ldw, scale, N, K, max_batch=1, flags=0, stream=None) -> int:
    h = ctypes.c_void_p()
    _check(lib().spike_proj_plan(ctypes.byref(h), _addr(W), ldw, _addr(scale), N, K,
                                 max_batch, flags, _stream(stream)), "spike_proj_plan")
    return h.value


def spike_proj_plan_destroy(plan):
    _check(lib().spike_proj_plan_destroy(plan), "spike_proj_plan_destroy")


def spike_proj_decode(plan, spikes, fmt, acc=None, y=None, stream=None):
    _check(lib().spike_proj_decode(plan, _addr(spikes), _fmt(fmt), _addr(acc), _addr(y),
                                   _stream(stream)), "spike_proj_decode")


def spike_proj_batched(plan, spikes, fmt, B, ld_spikes, acc=None, y=None, strategy="auto",
                       stream=None):
    _check(lib().spike_proj_batched(plan, _addr(spikes), _fmt(fmt), B, ld_spikes, _addr(acc),
                                    _addr(y), _kernel(strategy), _stream(stream)),
           "spike_proj_batched")


def spike_proj_prefill(plan, X, T, ldx, acc=None, y=None, strategy="auto", stream=None):
    _check(lib().spike_proj_prefill(plan, _addr(X), T, ldx, _addr(acc), _addr(y),
                                    _kernel(strategy), _stream(stream)), "spike_proj_prefill")


def spike_proj_last_dispatch(plan):
    k = ctypes.c_int(0)
    n = ctypes.c_int32(0)
    _check(lib().spike_proj_last_dispatch(plan, ctypes.byref(k), ctypes.byref(n)),
           "spike_proj_last_dispatch")
    return KERNEL_NAMES.get(k.value, k.value), n.value


def spike_proj_plan_status(plan, stream=None) -> int:
    return lib().spike_proj_plan_status(plan, _stream(stream))


def spike_proj_group_create(plans, stream=None) -> int:
    arr = (ctypes.c_void_p * len(plans))(*plans)
    h = ctypes.c_void_p()
    _check(lib().spike_proj_group_create(ctypes.byref(h), arr, len(plans), _stream(stream)),
           "spike_proj_group_create")
    return h.value


def spike_proj_group_destroy(group):
    _check(lib().spike_proj_group_destroy(group), "spike_proj_group_destroy")


def spike_proj_group_decode(group, spikes, fmt, ld_spikes, acc=None, y=None, ld_out=0,
                            stream=None):
    _check(lib().spike_proj_group_decode(group, _addr(spikes), _fmt(fmt), ld_spikes, _addr(acc),
                                         _addr(y), ld_out, _stream(stream)),
           "spike_proj_group_decode")


def spike_proj_group_decode_host(group, h_spikes, fmt, ld_spikes, h_acc=None, h_y=None,
                                 ld_out=0, stream=None):
    _check(lib().spike_proj_group_decode_host(group, _addr(h_spikes), _fmt(fmt), ld_spikes,
                                              _addr(h_acc), _addr(h_y), ld_out,
                                              _stream(stream)),
           "spike_proj_group_decode_host")


def spike_proj_group_decode_lif(group, v_in, v_out, I, ld, beta, theta, bits=None, ld_bits=0,
                                acc=None, y=None, ld_out=0, stream=None):
    _check(lib().spike_proj_group_decode_lif(group, _addr(v_in), _addr(v_out), _addr(I), ld, beta,
                                             theta, _addr(bits), ld_bits, _addr(acc), _addr(y),
                                             ld_out, _stream(stream)),
           "spike_proj_group_decode_lif")


def _ptr_array(xs):
    """Host array of device addresses (ctypes), or None."""
    if xs is None:
        return None
    return (ctypes.c_void_p * len(xs))(*[_addr(x) for x in xs])


def spike_proj_group_prefill(group, X, fmt, T, ldx, acc=None, y=None, stream=None):
    """X, acc, y: sequences with one device tensor (or address) per member."""
    _check(lib().spike_proj_group_prefill(group, _ptr_array(X), _fmt(fmt), T, ldx,
                                          _ptr_array(acc), _ptr_array(y), _stream(stream)),
           "spike_proj_group_prefill")


def spike_proj_group_status(group, stream=None) -> int:
    return lib().spike_proj_group_status(group, _stream(stream))


def spike_proj_lif(v, I, K, rows, ld, beta, theta, bits, ld_bits, stream=None):
    _check(lib().spike_proj_lif(_addr(v), _addr(I), K, rows, ld, beta, theta, _addr(bits), ld_bits,
                                _stream(stream)), "spike_proj_lif")


def lif(v, I, beta, theta, bits, K=None, stream=None):
    """One LIF step of every row of v / I (float32 [rows, ld] tensors),
    spikes into bits (uint32 [rows, >= ceil(K/32)])."""
    rows, ld = v.shape
    spike_proj_lif(v, I, ld if K is None else K, rows, v.stride(0), beta, theta, bits,
                   bits.stride(0), stream)


class SpDense(ctypes.Structure):
    """struct sp_dense of spike_proj.h (one continuous-input projection)."""
    _fields_ = [("W", ctypes.c_void_p), ("ldw", ctypes.c_int64), ("scale", ctypes.c_void_p),
                ("x", ctypes.c_void_p), ("ldx", ctypes.c_int64), ("y", ctypes.c_void_p),
                ("ldy", ctypes.c_int64), ("N", ctypes.c_int32), ("K", ctypes.c_int32)]


def spike_proj_dense(problems, B, stream=None):
    """problems: sequence of (W, ldw, scale, x, ldx, y, ldy, N, K), the fields
    of struct sp_dense (tensors or addresses); all run in one launch."""
    arr = (SpDense * len(problems))()
    for i, (W, ldw, scale, x, ldx, y, ldy, N, K) in enumerate(problems):
        arr[i] = SpDense(_addr(W), ldw, _addr(scale), _addr(x), ldx, _addr(y), ldy, N, K)
    _check(lib().spike_proj_dense(ctypes.addressof(arr), len(problems), B, _stream(stream)),
           "spike_proj_dense")


def dense(W, scale, x, y, K=None, stream=None):
    """One continuous-input projection: W int8 [N, ldw] row-major, scale
    float32 [N], x float32 [B, ldx], y float32 [B, ldy] (torch tensors)."""
    N, ldw = W.shape
    xs = x if x.dim() == 2 else x.reshape(1, -1)
    ys = y if y.dim() == 2 else y.reshape(1, -1)
    K = ldw if K is None else K
    spike_proj_dense([(W, ldw, scale, xs, xs.stride(0), ys, ys.stride(0), N, K)], xs.shape[0],
                     stream)


def spike_proj_decode_noalloc(W, ldw, scale, N, K, spikes, fmt, acc=None, y=None,
                              stream=None):
    """Batch-1 decode without a plan and without any allocation (the
    library's fixed per-device scratch; N <= SPIKE_PROJ_NOALLOC_MAX_N)."""
    _check(lib().spike_proj_decode_noalloc(_addr(W), ldw, _addr(scale), N, K, _addr(spikes),
                                           _fmt(fmt), _addr(acc), _addr(y), _stream(stream)),
           "spike_proj_decode_noalloc")


def spike_proj_probe_gather(base, offsets16, count, sink, piece_bytes=512, stream=None):
    """Measurement aid: read `count` pieces of `piece_bytes` at base + 16 * offsets16[i]."""
    _check(lib().spike_proj_probe_gather(_addr(base), _addr(offsets16), count, piece_bytes,
                                         _addr(sink), _stream(stream)), "spike_proj_probe_gather")


def spike_proj_plan_inject_fault(plan, fault):
    """Tests of the error path only: arm a fault for the plan's next launch."""
    _check(lib().spike_proj_plan_inject_fault(plan, fault), "spike_proj_plan_inject_fault")


def spike_proj_group_inject_fault(group, fault):
    """Tests of the error path only: arm a fault for the group's next launch."""
    _check(lib().spike_proj_group_inject_fault(group, fault), "spike_proj_group_inject_fault")


def spike_proj_strerror(status) -> str:
    return lib().spike_proj_strerror(status).decode()


def spike_proj_abi_version() -> int:
    return lib().spike_proj_abi_version()


# ---------------------------------------------------------------------------
# convenience owners (hold references to the borrowed tensors)
# ---------------------------------------------------------------------------
class Plan:
    """One projection: column-major INT8 W (torch int8 CUDA tensor whose
    storage is [K][ldw]) and FP32 scale [N]."""

    def __init__(self, W, scale, N, K, ldw=None, max_batch=1, gemm=False, stream=None):
        self.W, self.scale = W, scale            # borrowed by the library
        self.N, self.K = N, K
        self.ldw = N if ldw is None else ldw
        self.max_batch = max_batch
        self.handle = spike_proj_plan(W, self.ldw, scale, N, K, max_batch,
                                      SP_PLAN_GEMM if gemm else 0, stream)

    def decode(self, spikes, fmt, acc=None, y=None, stream=None):
        spike_proj_decode(self.handle, spikes, fmt, acc, y, stream)

    def batched(self, spikes, fmt, B, ld_spikes, acc=None, y=None, strategy="auto",
                stream=None):
        spike_proj_batched(self.handle, spikes, fmt, B, ld_spikes, acc, y, strategy, stream)

    def prefill(self, X, T, ldx, acc=None, y=None, strategy="auto", stream=None):
        spike_proj_prefill(self.handle, X, T, ldx, acc, y, strategy, stream)

    def last_dispatch(self):
        return spike_proj_last_dispatch(self.handle)

    def status(self, stream=None) -> int:
        return spike_proj_plan_status(self.handle, stream)

    def inject_fault(self, fault):
        """Tests of the error path only (SP_FAULT_ABORT / SP_FAULT_STALL)."""
        spike_proj_plan_inject_fault(self.handle, fault)

    def close(self):
        if self.handle:
            spike_proj_plan_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class Group:
    """Independent batch-1 projections decoded in one launch."""

    def __init__(self, plans, stream=None):
        self.plans = list(plans)
        self.handle = spike_proj_group_create([p.handle for p in self.plans], stream)

    def decode(self, spikes, fmt, ld_spikes, acc=None, y=None, ld_out=0, stream=None):
        spike_proj_group_decode(self.handle, spikes, fmt, ld_spikes, acc, y, ld_out, stream)

    def decode_host(self, h_spikes, fmt, ld_spikes, h_acc=None, h_y=None, ld_out=0,
                    stream=None):
        spike_proj_group_decode_host(self.handle, h_spikes, fmt, ld_spikes, h_acc, h_y,
                                     ld_out, stream)

    def decode_lif(self, v_in, v_out, I, beta, theta, bits=None, acc=None, y=None, ld_out=0,
                   stream=None):
        """One LIF step of row j of v_in / I (float32 [count, ld] tensors) into
        v_out, its spikes projected by plan j, in one launch; bits (uint32
        [count, >= ceil(maxK/32)]) optionally receives the spike words."""
        spike_proj_group_decode_lif(self.handle, v_in, v_out, I, v_in.stride(0), beta, theta, bits,
                                    0 if bits is None else bits.stride(0), acc, y, ld_out, stream)

    def prefill(self, X, fmt, T, ldx, acc=None, y=None, stream=None):
        """T rows per member through the tensor-core contraction, all members
        in one launch: X, acc, y hold one device tensor per member."""
        spike_proj_group_prefill(self.handle, X, fmt, T, ldx, acc, y, stream)

    def status(self, stream=None) -> int:
        return spike_proj_group_status(self.handle, stream)

    def inject_fault(self, fault):
        """Tests of the error path only (SP_FAULT_ABORT)."""
        spike_proj_group_inject_fault(self.handle, fault)

    def close(self):
        if self.handle:
            spike_proj_group_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def spike_proj_head_create(W, ldw, scale, V, K, stream=None) -> int:
    h = ctypes.c_void_p()
    _check(lib().spike_proj_head_create(ctypes.byref(h), _addr(W), ldw, _addr(scale), V, K,
                                        _stream(stream)), "spike_proj_head_create")
    return h.value


def spike_proj_head_destroy(head):
    _check(lib().spike_proj_head_destroy(head), "spike_proj_head_destroy")


def spike_proj_head(head, h, ldh, B, tau, k_sel, token, verified=None, gap=None, cand=None, r=None,
                    z=None, ld_z=0, stream=None):
    _check(lib().spike_proj_head(head, _addr(h), ldh, B, tau, k_sel, _addr(token), _addr(verified),
                                 _addr(gap), _addr(cand), _addr(r), _addr(z), ld_z,
                                 _stream(stream)), "spike_proj_head")


class Head:
    """Vocabulary head with INT8 activations and candidate-row verification
    over row-major INT8 weights W [V, ldw] and row scales [V] (borrowed)."""

    def __init__(self, W, scale, K=None, stream=None):
        self.W, self.scale = W, scale
        self.V, self.ldw = W.shape
        self.K = self.ldw if K is None else K
        self.handle = spike_proj_head_create(W, self.ldw, scale, self.V, self.K, stream)

    def __call__(self, h, tau, k_sel, token, verified=None, gap=None, cand=None, r=None, z=None,
                 stream=None):
        """h float32 [B, ldh]; outputs as spike_proj_head (tensors)."""
        hs = h if h.dim() == 2 else h.reshape(1, -1)
        spike_proj_head(self.handle, hs, hs.stride(0), hs.shape[0], tau, k_sel, token, verified,
                        gap, cand, r, z, 0 if z is None else z.stride(0), stream)

    def close(self):
        if self.handle:
            spike_proj_head_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
