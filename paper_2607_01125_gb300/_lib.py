"""ctypes binding of libzoact (include/zoact.h): argument marshalling only.

Every function below has the name of the C entry point it calls and passes
torch tensors as raw device pointers; no step of the ZO-Act path runs in
Python.  Loading fails loudly when the library has not been built: there is no
CPU fallback.
"""
import ctypes
import os

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libzoact.so")

ZOACT_OK = 0
ZOACT_ERR_INVALID_ARG = -1
ZOACT_ERR_UNSUPPORTED = -2
ZOACT_ERR_CUDA = -3
ZOACT_ERR_NONFINITE = -4
ZOACT_ERR_TIMEOUT = -5
ZOACT_ERR_NOMEM = -6
ZOACT_ERR_TOO_LARGE = -7
ZOACT_ERR_REPLICA_MISMATCH = -8
NOALLOC_MAX_PROJ_FLOATS = 1 << 20
MAX_EVAL_BLOCKS = 17
MAX_GROUP = 4

DT_FP32, DT_BF16, DT_FP16, DT_INT4_G128 = 0, 1, 2, 3
ACT_NONE, ACT_RELU, ACT_GELU = 0, 1, 2

TORCH_DT = {torch.float32: DT_FP32, torch.bfloat16: DT_BF16, torch.float16: DT_FP16}

# every entry point include/zoact.h declares
EXPORTS = [
    "zoact_create", "zoact_destroy", "zoact_set_stream", "zoact_status_string", "zoact_get_device_status",
    "zoact_device_sm_count", "zoact_get_launch_count", "zoact_philox_normals", "zoact_lowrank_proj", "zoact_pair_forward",
    "zoact_pair_forward_noalloc", "zoact_pair_forward_gated", "zoact_loss_pair", "zoact_adam_step", "zoact_sgd_step", "zoact_basis_init",
    "zoact_rms_norm", "zoact_mix_rms", "zoact_multi_forward", "zoact_multi_forward_gated", "zoact_loss_multi",
    "zoact_adam_step_multi", "zoact_sgd_step_multi", "zoact_basis_prepared_bytes", "zoact_basis_prepare",
    "zoact_lowrank_proj_prepared", "zoact_subspace_overlap", "zoact_gradient_energy", "zoact_kernel_timing",
    "zoact_kernel_time", "zoact_pair_forward_loss", "zoact_debug_timeout", "zoact_mean_over_ranks",
    "zoact_arena_hash", "zoact_pair_forward_rs", "zoact_pair_forward_gated_rs", "zoact_rms_scale",
    "zoact_multi_forward_rs", "zoact_multi_forward_gated_rs", "zoact_pair_forward_group_rs",
    "zoact_multi_forward_group_rs", "zoact_mix_rms_strided",
]


class ZoactError(RuntimeError):
    def __init__(self, fn, status):
        self.status = status
        super().__init__(f"{fn} failed: {status} ({status_string(status)})")


class zoact_layer(ctypes.Structure):
    _fields_ = [("d_in", ctypes.c_int32), ("d_out", ctypes.c_int32), ("r", ctypes.c_int32),
                ("wtype", ctypes.c_int32), ("W", ctypes.c_void_p), ("w_scales", ctypes.c_void_p),
                ("U", ctypes.c_void_p), ("C", ctypes.c_void_p), ("layer_id", ctypes.c_uint32)]


class zoact_coeff_block(ctypes.Structure):
    _fields_ = [("offset", ctypes.c_int64), ("d_out", ctypes.c_int32), ("r", ctypes.c_int32),
                ("layer_id", ctypes.c_uint32), ("reserved", ctypes.c_uint32)]


class zoact_rowscale(ctypes.Structure):
    _fields_ = [("in_scale", ctypes.c_void_p), ("out_sumsq", ctypes.c_void_p)]


class zoact_eval_blocks(ctypes.Structure):
    _fields_ = [("n_blocks", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("coef", ctypes.c_float * MAX_EVAL_BLOCKS), ("query", ctypes.c_uint64 * MAX_EVAL_BLOCKS)]


def eval_blocks(points):
    """A zoact_eval_blocks from a list of (coef, query) pairs (block order = row-block order)."""
    if not 1 <= len(points) <= MAX_EVAL_BLOCKS:
        raise ValueError(f"1 .. {MAX_EVAL_BLOCKS} evaluation blocks")
    b = zoact_eval_blocks(n_blocks=len(points))
    for i, (c, q) in enumerate(points):
        b.coef[i] = float(c)
        b.query[i] = int(q)
    return b


def one_sided_blocks(mu, queries):
    """Algorithm 2's evaluation points: the unperturbed pass, then C + mu Z^(j) for each query."""
    return [(0.0, 0)] + [(float(mu), int(q)) for q in queries]


_lib = None


def load():
    """Load libzoact.so (built in-tree by __graft_entry__.build())."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"libzoact.so is not built ({LIB_PATH}); run __graft_entry__.build()")
    lib = ctypes.CDLL(LIB_PATH)
    P, I32, I64, U32, U64, F32 = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32,
                                  ctypes.c_uint64, ctypes.c_float)
    sig = {
        "zoact_create": [ctypes.POINTER(ctypes.c_void_p), I32, P],
        "zoact_destroy": [P],
        "zoact_set_stream": [P, P],
        "zoact_get_device_status": [P, ctypes.POINTER(ctypes.c_int), I32],
        "zoact_device_sm_count": [P, ctypes.POINTER(ctypes.c_int)],
        "zoact_get_launch_count": [P, ctypes.POINTER(ctypes.c_int64)],
        "zoact_debug_timeout": [P, I64],
        "zoact_philox_normals": [P, U64, U32, U64, I64, P, P],
        "zoact_lowrank_proj": [P, P, I32, I64, I32, P, I32, P],
        "zoact_pair_forward": [P, ctypes.POINTER(zoact_layer), P, I32, I64, I32, P, F32, U64, U64, I32, P, I32],
        "zoact_pair_forward_noalloc": [ctypes.POINTER(zoact_layer), P, I32, I64, I32, F32, U64, U64, I32, P, I32, P],
        "zoact_pair_forward_gated": [P, ctypes.POINTER(zoact_layer), ctypes.POINTER(zoact_layer), P, I32, I64, I32,
                                     P, P, F32, U64, U64, P, I32],
        "zoact_pair_forward_loss": [P, ctypes.POINTER(zoact_layer), P, I32, I64, P, F32, U64, U64, I32, I32, P, P],
        "zoact_loss_pair": [P, P, I32, P, I64, I64, F32, P],
        "zoact_adam_step": [P, P, P, P, I64, ctypes.POINTER(zoact_coeff_block), I32, P, F32, F32, F32, F32, I64,
                            U64, U64],
        "zoact_sgd_step": [P, P, I64, ctypes.POINTER(zoact_coeff_block), I32, P, F32, U64, U64],
        "zoact_basis_init": [P, P, I32, I64, I32, I32, I32, I32, U64, P, P],
        "zoact_rms_norm": [P, P, I32, I64, I32, F32, P],
        "zoact_mix_rms": [P, P, P, P, I32, I64, I32, I32, I32, F32, P],
        "zoact_basis_prepare": [P, P, I32, I32, I32, P],
        "zoact_lowrank_proj_prepared": [P, P, I32, I64, I32, P, I32, P],
        "zoact_kernel_timing": [P, I32],
        "zoact_kernel_time": [P, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_int64)],
        "zoact_subspace_overlap": [P, P, P, I32, I32, I32, P],
        "zoact_gradient_energy": [P, P, I32, I32, P, I32, I64, P],
        "zoact_multi_forward": [P, ctypes.POINTER(zoact_layer), P, I32, I64, I32, P, ctypes.POINTER(zoact_eval_blocks),
                                U64, I32, P, I32],
        "zoact_multi_forward_gated": [P, ctypes.POINTER(zoact_layer), ctypes.POINTER(zoact_layer), P, I32, I64, I32,
                                      P, P, ctypes.POINTER(zoact_eval_blocks), U64, P, I32],
        "zoact_loss_multi": [P, P, I32, P, I64, I64, I32, F32, P],
        "zoact_adam_step_multi": [P, P, P, P, I64, ctypes.POINTER(zoact_coeff_block), I32, P, I32,
                                  ctypes.POINTER(ctypes.c_uint64), F32, F32, F32, F32, I64, U64],
        "zoact_sgd_step_multi": [P, P, I64, ctypes.POINTER(zoact_coeff_block), I32, P, I32,
                                 ctypes.POINTER(ctypes.c_uint64), F32, U64],
        "zoact_mean_over_ranks": [P, P, I64, I32],
        "zoact_pair_forward_rs": [P, ctypes.POINTER(zoact_layer), P, I32, I64, I32, P, F32, U64, U64, I32, P, I32,
                                  ctypes.POINTER(zoact_rowscale)],
        "zoact_pair_forward_gated_rs": [P, ctypes.POINTER(zoact_layer), ctypes.POINTER(zoact_layer), P, I32, I64, I32,
                                        P, P, F32, U64, U64, P, I32, ctypes.POINTER(zoact_rowscale)],
        "zoact_rms_scale": [P, P, I64, I32, F32, P],
        "zoact_multi_forward_rs": [P, ctypes.POINTER(zoact_layer), P, I32, I64, I32, P,
                                   ctypes.POINTER(zoact_eval_blocks), U64, I32, P, I32, ctypes.POINTER(zoact_rowscale)],
        "zoact_multi_forward_gated_rs": [P, ctypes.POINTER(zoact_layer), ctypes.POINTER(zoact_layer), P, I32, I64, I32,
                                         P, P, ctypes.POINTER(zoact_eval_blocks), U64, P, I32,
                                         ctypes.POINTER(zoact_rowscale)],
        "zoact_arena_hash": [P, P, I64, P],
        "zoact_pair_forward_group_rs": [P, ctypes.POINTER(zoact_layer), I32, P, I32, I64, P, F32, U64, U64, I32, P,
                                        I32, ctypes.POINTER(zoact_rowscale)],
        "zoact_multi_forward_group_rs": [P, ctypes.POINTER(zoact_layer), I32, P, I32, I64, P,
                                         ctypes.POINTER(zoact_eval_blocks), U64, I32, P, I32,
                                         ctypes.POINTER(zoact_rowscale)],
        "zoact_mix_rms_strided": [P, P, P, P, I32, I64, I32, I32, I32, I64, I64, F32, P],
    }
    for name, argtypes in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = argtypes
        fn.restype = ctypes.c_int
    lib.zoact_basis_prepared_bytes.argtypes = [I32, I32]
    lib.zoact_basis_prepared_bytes.restype = ctypes.c_int64
    lib.zoact_status_string.argtypes = [ctypes.c_int]
    lib.zoact_status_string.restype = ctypes.c_char_p
    _lib = lib
    return lib


def status_string(status):
    return load().zoact_status_string(int(status)).decode()


def _check(name, status):
    if status != ZOACT_OK:
        raise ZoactError(name, status)


def _ptr(t):
    """Device address of a row-major tensor (the ABI's layout); other layouts are refused."""
    if t is None:
        return None
    if not t.is_contiguous():
        raise ValueError("libzoact takes row-major (contiguous) tensors")
    return ctypes.c_void_p(t.data_ptr())


def _dt(t):
    return TORCH_DT[t.dtype]


class Context:
    """A libzoact context bound to one CUDA device; launches on torch's current stream."""

    def __init__(self, device=0):
        lib = load()
        self.device = int(device)
        h = ctypes.c_void_p()
        with torch.cuda.device(self.device):
            stream = torch.cuda.current_stream().cuda_stream
        _check("zoact_create", lib.zoact_create(ctypes.byref(h), self.device, ctypes.c_void_p(stream)))
        self.handle = h

    def sync_stream(self):
        """Point the context at torch's current stream on its device."""
        with torch.cuda.device(self.device):
            s = torch.cuda.current_stream().cuda_stream
        load().zoact_set_stream(self.handle, ctypes.c_void_p(s))

    def sm_count(self):
        v = ctypes.c_int()
        _check("zoact_device_sm_count", load().zoact_device_sm_count(self.handle, ctypes.byref(v)))
        return v.value

    def launch_count(self):
        v = ctypes.c_int64()
        _check("zoact_get_launch_count", load().zoact_get_launch_count(self.handle, ctypes.byref(v)))
        return v.value

    def kernel_timing(self, enable=True):
        """Record events around every tensor-core pair-forward kernel (see zoact_kernel_timing)."""
        _check("zoact_kernel_timing", load().zoact_kernel_timing(self.handle, int(enable)))

    def kernel_time(self):
        """(summed milliseconds, launches) of the timed pair-forward kernels since the last read; syncs."""
        ms, n = ctypes.c_double(), ctypes.c_int64()
        _check("zoact_kernel_time", load().zoact_kernel_time(self.handle, ctypes.byref(ms), ctypes.byref(n)))
        return ms.value, n.value

    def debug_timeout(self, wait_ns):
        """Failure-detection test hook (see zoact_debug_timeout): a bounded wait that runs out."""
        _check("zoact_debug_timeout", load().zoact_debug_timeout(self.handle, int(wait_ns)))

    def device_status(self, reset=True):
        v = ctypes.c_int()
        _check("zoact_get_device_status", load().zoact_get_device_status(self.handle, ctypes.byref(v), int(reset)))
        return v.value

    def close(self):
        if getattr(self, "handle", None):
            load().zoact_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def make_layer(W, U, C, layer_id, w_scales=None, wtype=None, d_in=None):
    """A zoact_layer for torch tensors W [d_out, d_in] (or INT4 packed), U [d_in, r] fp32, C [d_out, r] fp32."""
    for t in (W, U, C, w_scales):
        if t is not None and not t.is_contiguous():
            raise ValueError("libzoact takes row-major (contiguous) tensors")
    if wtype is None:
        wtype = _dt(W)
    d_out = W.shape[0]
    if d_in is None:
        d_in = W.shape[1] * (2 if wtype == DT_INT4_G128 else 1)
    L = zoact_layer(d_in=int(d_in), d_out=int(d_out), r=int(U.shape[1]), wtype=int(wtype),
                    W=W.data_ptr(), w_scales=(w_scales.data_ptr() if w_scales is not None else None),
                    U=U.data_ptr(), C=C.data_ptr(), layer_id=int(layer_id))
    L._keep = (W, U, C, w_scales)
    return L


def zoact_philox_normals(ctx, seed, layer_id, query, n, z_out, words_out=None):
    _check("zoact_philox_normals", load().zoact_philox_normals(ctx.handle, seed, layer_id, query, n, _ptr(z_out),
                                                                _ptr(words_out)))


def zoact_lowrank_proj(ctx, X, U, P):
    rows, d_in = X.shape
    _check("zoact_lowrank_proj", load().zoact_lowrank_proj(ctx.handle, _ptr(X), _dt(X), rows, d_in, _ptr(U),
                                                            U.shape[1], _ptr(P)))


def zoact_pair_forward(ctx, layer, X, T, input_shared, eps, seed, query, Y, P=None, act=ACT_NONE):
    _check("zoact_pair_forward", load().zoact_pair_forward(ctx.handle, ctypes.byref(layer), _ptr(X), _dt(X), int(T),
                                                            int(input_shared), _ptr(P), float(eps), int(seed),
                                                            int(query), int(act), _ptr(Y), _dt(Y)))


def zoact_pair_forward_noalloc(layer, X, T, input_shared, eps, seed, query, Y, act=ACT_NONE, stream=None):
    """The pair forward without a context or any device allocation (see include/zoact.h).

    For callers that cannot allocate device memory; scratch is a fixed static
    device array shared by all calls.  `stream` defaults to torch's current stream.
    """
    if stream is None:
        stream = torch.cuda.current_stream().cuda_stream
    _check("zoact_pair_forward_noalloc", load().zoact_pair_forward_noalloc(
        ctypes.byref(layer), _ptr(X), _dt(X), int(T), int(input_shared), float(eps), int(seed), int(query),
        int(act), _ptr(Y), _dt(Y), ctypes.c_void_p(stream)))


def zoact_pair_forward_gated(ctx, gate, up, X, T, input_shared, eps, seed, query, H, P_gate=None, P_up=None):
    _check("zoact_pair_forward_gated", load().zoact_pair_forward_gated(
        ctx.handle, ctypes.byref(gate), ctypes.byref(up), _ptr(X), _dt(X), int(T), int(input_shared), _ptr(P_gate),
        _ptr(P_up), float(eps), int(seed), int(query), _ptr(H), _dt(H)))


def zoact_pair_forward_loss(ctx, layer, X, T, eps, seed, query, ydtype, out, target=None, P=None, act=ACT_NONE):
    """The pair forward of `layer` on stacked X [2T, d_in] fused with its loss pair: out[4] = {L+, L-, D, a} of
    the outputs rounded to ydtype (DT_BF16 / DT_FP16), Y not written.  Raises ZoactError with status
    ZOACT_ERR_UNSUPPORTED when the launch does not qualify (see include/zoact.h)."""
    _check("zoact_pair_forward_loss", load().zoact_pair_forward_loss(
        ctx.handle, ctypes.byref(layer), _ptr(X), _dt(X), int(T), _ptr(P), float(eps), int(seed), int(query),
        int(act), int(ydtype), _ptr(target), _ptr(out)))


def zoact_loss_pair(ctx, Y, T, eps, out, target=None):
    n = Y.shape[1]
    _check("zoact_loss_pair", load().zoact_loss_pair(ctx.handle, _ptr(Y), _dt(Y), _ptr(target), int(T), int(n),
                                                      float(eps), _ptr(out)))


def _blocks(blocks):
    arr = (zoact_coeff_block * max(1, len(blocks)))()
    for i, (offset, d_out, r, layer_id) in enumerate(blocks):
        arr[i] = zoact_coeff_block(offset=int(offset), d_out=int(d_out), r=int(r), layer_id=int(layer_id))
    return arr


def zoact_adam_step(ctx, C, m, v, blocks, loss_out, lr, beta1, beta2, adam_eps, step, seed, query):
    """blocks: list of (offset, d_out, r, layer_id) into the flat arenas C, m, v."""
    arr = _blocks(blocks)
    _check("zoact_adam_step", load().zoact_adam_step(ctx.handle, _ptr(C), _ptr(m), _ptr(v), C.numel(), arr,
                                                      len(blocks), _ptr(loss_out), float(lr), float(beta1),
                                                      float(beta2), float(adam_eps), int(step), int(seed),
                                                      int(query)))


def zoact_sgd_step(ctx, C, blocks, loss_out, lr, seed, query):
    arr = _blocks(blocks)
    _check("zoact_sgd_step", load().zoact_sgd_step(ctx.handle, _ptr(C), C.numel(), arr, len(blocks),
                                                    _ptr(loss_out), float(lr), int(seed), int(query)))


def zoact_basis_init(ctx, X_cal, r, U_out, oversample=8, n_iter=8, seed=0, evals_out=None):
    n_tok, d_in = X_cal.shape
    _check("zoact_basis_init", load().zoact_basis_init(ctx.handle, _ptr(X_cal), _dt(X_cal), n_tok, d_in, int(r),
                                                        int(oversample), int(n_iter), int(seed), _ptr(U_out),
                                                        _ptr(evals_out)))


def zoact_rms_norm(ctx, X, Y, eps=1e-5):
    rows, n = X.shape
    _check("zoact_rms_norm", load().zoact_rms_norm(ctx.handle, _ptr(X), _dt(X), rows, n, float(eps), _ptr(Y)))


def zoact_mix_rms(ctx, q, k, v, Y, n_rep, head_dim, eps=1e-5):
    """Y = rms(q + rep(k) + rep(v)).  q, k and v may be column views (unit column stride) of wider row-major
    tensors -- the layers' columns of a zoact_pair_forward_group_rs output -- which go to zoact_mix_rms_strided."""
    rows, n = q.shape
    if q.is_contiguous() and k.is_contiguous() and v.is_contiguous():
        _check("zoact_mix_rms", load().zoact_mix_rms(ctx.handle, _ptr(q), _ptr(k), _ptr(v), _dt(q), rows, n,
                                                      int(n_rep), int(head_dim), float(eps), _ptr(Y)))
        return
    if q.stride(1) != 1 or k.stride(1) != 1 or v.stride(1) != 1 or k.stride(0) != v.stride(0):
        raise ValueError("libzoact takes rows with unit column stride (k and v with one row stride)")
    _check("zoact_mix_rms_strided", load().zoact_mix_rms_strided(
        ctx.handle, ctypes.c_void_p(q.data_ptr()), ctypes.c_void_p(k.data_ptr()), ctypes.c_void_p(v.data_ptr()),
        _dt(q), rows, n, int(n_rep), int(head_dim), int(q.stride(0)), int(k.stride(0)), float(eps), _ptr(Y)))


def zoact_multi_forward(ctx, layer, X, T, input_shared, points, seed, Y, P=None, act=ACT_NONE):
    """points: list of (coef, query); Y has len(points) * T rows."""
    b = eval_blocks(points)
    _check("zoact_multi_forward", load().zoact_multi_forward(ctx.handle, ctypes.byref(layer), _ptr(X), _dt(X), int(T),
                                                              int(input_shared), _ptr(P), ctypes.byref(b), int(seed),
                                                              int(act), _ptr(Y), _dt(Y)))


def zoact_multi_forward_gated(ctx, gate, up, X, T, input_shared, points, seed, H, P_gate=None, P_up=None):
    b = eval_blocks(points)
    _check("zoact_multi_forward_gated", load().zoact_multi_forward_gated(
        ctx.handle, ctypes.byref(gate), ctypes.byref(up), _ptr(X), _dt(X), int(T), int(input_shared), _ptr(P_gate),
        _ptr(P_up), ctypes.byref(b), int(seed), _ptr(H), _dt(H)))


def zoact_loss_multi(ctx, Y, T, n_blocks, mu, out, target=None):
    """out: device fp64 [2 n_blocks - 1] = [L_0 .. L_{nb-1}, a_1 .. a_q]."""
    n = Y.shape[1]
    _check("zoact_loss_multi", load().zoact_loss_multi(ctx.handle, _ptr(Y), _dt(Y), _ptr(target), int(T), int(n),
                                                        int(n_blocks), float(mu), _ptr(out)))


def _queries(queries):
    arr = (ctypes.c_uint64 * max(1, len(queries)))()
    for i, q in enumerate(queries):
        arr[i] = int(q)
    return arr


def zoact_adam_step_multi(ctx, C, m, v, blocks, a, queries, lr, beta1, beta2, adam_eps, step, seed):
    """a: device fp64 tensor of len(queries) estimator scalars (e.g. a slice of zoact_loss_multi's out)."""
    arr = _blocks(blocks)
    _check("zoact_adam_step_multi", load().zoact_adam_step_multi(
        ctx.handle, _ptr(C), _ptr(m), _ptr(v), C.numel(), arr, len(blocks), _ptr(a), len(queries),
        _queries(queries), float(lr), float(beta1), float(beta2), float(adam_eps), int(step), int(seed)))


def zoact_sgd_step_multi(ctx, C, blocks, a, queries, lr, seed):
    arr = _blocks(blocks)
    _check("zoact_sgd_step_multi", load().zoact_sgd_step_multi(ctx.handle, _ptr(C), C.numel(), arr, len(blocks),
                                                                _ptr(a), len(queries), _queries(queries), float(lr),
                                                                int(seed)))


def zoact_basis_prepared_bytes(d_in, r):
    return int(load().zoact_basis_prepared_bytes(int(d_in), int(r)))


def zoact_basis_prepare(ctx, U, xdtype, U_tc):
    """U [d_in, r] fp32 -> U_tc (uint8 device tensor of zoact_basis_prepared_bytes bytes) for X of xdtype."""
    d_in, r = U.shape
    _check("zoact_basis_prepare", load().zoact_basis_prepare(ctx.handle, _ptr(U), d_in, r, int(xdtype), _ptr(U_tc)))


def zoact_lowrank_proj_prepared(ctx, X, U_tc, r, P):
    rows, d_in = X.shape
    _check("zoact_lowrank_proj_prepared", load().zoact_lowrank_proj_prepared(ctx.handle, _ptr(X), _dt(X), rows, d_in,
                                                                              _ptr(U_tc), int(r), _ptr(P)))


def zoact_subspace_overlap(ctx, U_a, U_b, out):
    """out: device fp64 [3] = [||U_a^T U_b||^2, ||U_b||^2, ||U_a^T U_b||^2 / r_a]."""
    d, ra = U_a.shape
    _check("zoact_subspace_overlap", load().zoact_subspace_overlap(ctx.handle, _ptr(U_a), _ptr(U_b), d, ra,
                                                                    U_b.shape[1], _ptr(out)))


def zoact_gradient_energy(ctx, U, G, out):
    """out: device fp64 [3] = [||U^T G||^2, ||G||^2, ratio]; G [d_in, n]."""
    d_in, r = U.shape
    _check("zoact_gradient_energy", load().zoact_gradient_energy(ctx.handle, _ptr(U), d_in, r, _ptr(G), _dt(G),
                                                                  G.shape[1], _ptr(out)))


def zoact_mean_over_ranks(ctx, v, world):
    """v (device fp64) /= world in place: the all-reduced sum of the ranks' loss vectors -> their mean."""
    _check("zoact_mean_over_ranks", load().zoact_mean_over_ranks(ctx.handle, _ptr(v), v.numel(), int(world)))


def zoact_arena_hash(ctx, t, out):
    """The 64-bit fingerprint of t's bytes (a device tensor whose size is a multiple of 4 bytes) written to
    out (a device int64 tensor of one element holding the uint64's bits)."""
    nbytes = t.numel() * t.element_size()
    if nbytes % 4 or out.dtype != torch.int64 or out.numel() != 1:
        raise ValueError("zoact_arena_hash: a tensor of whole 32-bit words and a one-element int64 output")
    _check("zoact_arena_hash", load().zoact_arena_hash(ctx.handle, _ptr(t), nbytes // 4, _ptr(out)))


def rowscale_parts(d_out):
    """Rows of the out_sumsq array a pair forward with row scales writes for d_out output columns."""
    return (int(d_out) + 63) // 64


def _rowscale(in_scale, out_sumsq):
    return zoact_rowscale(in_scale=None if in_scale is None else _ptr(in_scale).value,
                          out_sumsq=None if out_sumsq is None else _ptr(out_sumsq).value)


def zoact_pair_forward_rs(ctx, layer, X, T, input_shared, eps, seed, query, Y, P=None, act=ACT_NONE, in_scale=None,
                          out_sumsq=None):
    """zoact_pair_forward with row scales (see include/zoact.h); raises ZoactError with ZOACT_ERR_UNSUPPORTED
    where the launch cannot apply them."""
    rs = _rowscale(in_scale, out_sumsq)
    _check("zoact_pair_forward_rs", load().zoact_pair_forward_rs(
        ctx.handle, ctypes.byref(layer), _ptr(X), _dt(X), int(T), int(input_shared), _ptr(P), float(eps), int(seed),
        int(query), int(act), _ptr(Y), _dt(Y), ctypes.byref(rs)))


def zoact_pair_forward_gated_rs(ctx, gate, up, X, T, input_shared, eps, seed, query, H, P_gate=None, P_up=None,
                                in_scale=None, out_sumsq=None):
    rs = _rowscale(in_scale, out_sumsq)
    _check("zoact_pair_forward_gated_rs", load().zoact_pair_forward_gated_rs(
        ctx.handle, ctypes.byref(gate), ctypes.byref(up), _ptr(X), _dt(X), int(T), int(input_shared), _ptr(P_gate),
        _ptr(P_up), float(eps), int(seed), int(query), _ptr(H), _dt(H), ctypes.byref(rs)))


def zoact_rms_scale(ctx, sumsq, n, inv_scale, eps=1e-5):
    """inv_scale [rows] = 1 / sqrt(sum_p sumsq[p] / n + eps) for sumsq [rowscale_parts(n), rows]."""
    rows = sumsq.shape[-1]
    _check("zoact_rms_scale", load().zoact_rms_scale(ctx.handle, _ptr(sumsq), int(rows), int(n), float(eps),
                                                      _ptr(inv_scale)))


def zoact_multi_forward_rs(ctx, layer, X, T, input_shared, points, seed, Y, P=None, act=ACT_NONE, in_scale=None,
                           out_sumsq=None):
    """zoact_multi_forward with row scales (see include/zoact.h)."""
    b = eval_blocks(points)
    rs = _rowscale(in_scale, out_sumsq)
    _check("zoact_multi_forward_rs", load().zoact_multi_forward_rs(
        ctx.handle, ctypes.byref(layer), _ptr(X), _dt(X), int(T), int(input_shared), _ptr(P), ctypes.byref(b),
        int(seed), int(act), _ptr(Y), _dt(Y), ctypes.byref(rs)))


def _layer_array(layers):
    if not 1 <= len(layers) <= MAX_GROUP:
        raise ValueError(f"1 .. {MAX_GROUP} layers per group")
    arr = (zoact_layer * len(layers))()
    for i, l in enumerate(layers):
        ctypes.memmove(ctypes.byref(arr[i]), ctypes.byref(l), ctypes.sizeof(zoact_layer))
    return arr


def zoact_pair_forward_group_rs(ctx, layers, X, T, eps, seed, query, Y, P=None, act=ACT_NONE, in_scale=None,
                                out_sumsq=None):
    """Layers that read X (stacked rows), with contiguous weights and one basis, as one pair forward: Y
    [2T, sum d_out] holds their outputs side by side (include/zoact.h).  Raises ZoactError with
    ZOACT_ERR_UNSUPPORTED, before anything is launched, where one launch cannot serve them."""
    arr = _layer_array(layers)
    rs = _rowscale(in_scale, out_sumsq)
    _check("zoact_pair_forward_group_rs", load().zoact_pair_forward_group_rs(
        ctx.handle, arr, len(layers), _ptr(X), _dt(X), int(T), _ptr(P), float(eps), int(seed), int(query), int(act),
        _ptr(Y), _dt(Y), ctypes.byref(rs)))


def zoact_multi_forward_group_rs(ctx, layers, X, T, points, seed, Y, P=None, act=ACT_NONE, in_scale=None,
                                 out_sumsq=None):
    """zoact_pair_forward_group_rs over the evaluation blocks `points` (list of (coef, query))."""
    arr = _layer_array(layers)
    b = eval_blocks(points)
    rs = _rowscale(in_scale, out_sumsq)
    _check("zoact_multi_forward_group_rs", load().zoact_multi_forward_group_rs(
        ctx.handle, arr, len(layers), _ptr(X), _dt(X), int(T), _ptr(P), ctypes.byref(b), int(seed), int(act),
        _ptr(Y), _dt(Y), ctypes.byref(rs)))


def zoact_multi_forward_gated_rs(ctx, gate, up, X, T, input_shared, points, seed, H, P_gate=None, P_up=None,
                                 in_scale=None, out_sumsq=None):
    b = eval_blocks(points)
    rs = _rowscale(in_scale, out_sumsq)
    _check("zoact_multi_forward_gated_rs", load().zoact_multi_forward_gated_rs(
        ctx.handle, ctypes.byref(gate), ctypes.byref(up), _ptr(X), _dt(X), int(T), int(input_shared), _ptr(P_gate),
        _ptr(P_up), ctypes.byref(b), int(seed), _ptr(H), _dt(H), ctypes.byref(rs)))
