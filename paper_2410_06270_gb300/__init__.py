"""Python binding of libmc.so, the GB300 (sm_103a) C-ABI library for the compressed
MoE layer of "MC: Mixture Compressor for MoE LLMs" (PMQ mixed-bit experts, ODP).

Argument marshalling only: every step of the layer runs in the library's CUDA
kernels.  Functions carry the C names without the ``mc_`` prefix; tensors are
torch tensors on the current CUDA device and work is enqueued on torch's current
stream.  If the library has not been built, importing this package raises.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libmc.so")

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_CUDA, ERR_TIMEOUT, ERR_BAD_PACK, ERR_RANGE = 0, -1, -2, -3, -4, -5, -6

PATH_AUTO, PATH_GEMV, PATH_GEMM = 0, 1, 2


class MCError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__("mc error %d: %s" % (code, msg))
        self.code = code


class Shape(ctypes.Structure):
    _fields_ = [("E", ctypes.c_int32), ("H", ctypes.c_int32), ("F", ctypes.c_int32),
                ("group", ctypes.c_int32), ("top_k", ctypes.c_int32)]

    def __init__(self, E, H, F, group, top_k=2):
        super().__init__(E, H, F, group, top_k)


_lib = None


def load():
    """Load libmc.so; raises ImportError if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise ImportError("libmc.so not built: run `python -c 'import __graft_entry__ as g; g.build()'` "
                          "or `python paper_2410_06270_gb300/build.py`")
    lib = ctypes.CDLL(LIB_PATH)
    P, I, Z, F32 = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t, ctypes.c_float
    S = ctypes.POINTER(Shape)
    sig = {
        "mc_last_error": (ctypes.c_char_p, []),
        "mc_version": (I, []),
        "mc_pack_format_version": (I, []),
        "mc_packed_size": (Z, [S, P]),
        "mc_pack_experts_host": (I, [S, P, P, P, P, P, Z]),
        "mc_pack_experts": (I, [S, P, P, P, P, P, Z, P]),
        "mc_unpack_experts_host": (I, [P, Z, I, I, P, P, P]),
        "mc_unpack_experts": (I, [S, P, P, I, I, P, P, P, P, P]),
        "mc_pack_verify": (I, [S, P, P, Z]),
        "mc_route": (I, [P, P, I, S, F32, P, P, P, P, P, P, P]),
        "mc_moe_workspace_size": (Z, [S, I]),
        "mc_moe_forward": (I, [P, P, I, S, P, P, F32, P, P, P, Z, P, P, P, P]),
        "mc_moe_forward_static": (I, [P, P, I, S, P, P, F32, P, P, P, P]),
        "mc_stack_workspace_size": (Z, [S, I]),
        "mc_stack_forward": (I, [P, I, S, I, P, P, P, P, P, P, F32, P, Z, P]),
        "mc_set_path": (I, [I]),
        "mc_set_debug": (I, [I, ctypes.c_ulonglong]),
        "mc_check_status": (I, [P, P]),
        "mc_rmsnorm": (I, [P, P, I, I, F32, P, P]),
        "mc_add": (I, [P, P, Z, P, P]),
        "mc_selftest_umma": (I, [P, P, P, I, I, P, P]),
        "mc_token_importance_workspace_size": (Z, [I]),
        "mc_token_importance": (I, [P, P, I, I, I, F32, P, P, P, Z, P]),
        "mc_odp_threshold_host": (I, [P, P, I, ctypes.c_double, P]),
        "mc_expert_significance_host": (I, [P, P, P, I, I, P, P]),
        "mc_pmq_allocate": (I, [P, P, P, I, I, ctypes.c_double, ctypes.c_double, ctypes.c_double, P, P]),
        "mc_profile_enable": (I, [I]),
        "mc_profile_select": (ctypes.c_uint, [ctypes.c_uint]),
        "mc_profile_read": (I, [P, P, I]),
        "mc_profile_clear": (I, []),
        "mc_profile_name": (ctypes.c_char_p, [I]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def last_error() -> str:
    return load().mc_last_error().decode()


def _check(rc):
    if rc != OK:
        raise MCError(rc, last_error())


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


def _stream():
    import torch
    return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)


def _bits(bits):
    return np.ascontiguousarray(bits, dtype=np.int8)


class _PtrArray:
    """A C array of host pointers to numpy buffers (kept alive with it)."""

    def __init__(self, arrs):
        self.arrs = arrs
        self.arr = (ctypes.c_void_p * len(arrs))(*[None if a is None else a.ctypes.data for a in arrs])

    @property
    def as_parameter(self):
        return ctypes.cast(self.arr, ctypes.c_void_p)


def _ptr_array(arrs, ctype=None):
    return _PtrArray(arrs).as_parameter


def version() -> int:
    return load().mc_version()


# ------------------------------------------------------------------ packing --

def packed_size(shape: Shape, bits) -> int:
    b = _bits(bits)
    n = load().mc_packed_size(ctypes.byref(shape), b.ctypes.data)
    if n == 0:
        raise MCError(ERR_INVALID_ARG, last_error())
    return n


def _canon(codes, scales, zeros, bits=None):
    """Host arrays for the pack entry points: uint8 codes and fp16 scale / zero;
    a 16-bit expert's codes are its fp16 weights and its scale / zero are None."""
    dense = [bits is not None and int(bits[i // 3]) == 16 for i in range(len(codes))]
    c = [np.ascontiguousarray(np.asarray(a, dtype=np.float16)).view(np.uint16) if d
         else np.ascontiguousarray(a, dtype=np.uint8) for a, d in zip(codes, dense)]
    s = [None if d else np.ascontiguousarray(np.asarray(a, dtype=np.float16)).view(np.uint16)
         for a, d in zip(scales, dense)]
    z = [None if d else np.ascontiguousarray(np.asarray(a, dtype=np.float16)).view(np.uint16)
         for a, d in zip(zeros, dense)]
    return c, s, z


def pack_experts_host(shape: Shape, bits, codes, scales, zeros) -> np.ndarray:
    """codes/scales/zeros: flat lists of 3*E arrays indexed [3*e + m]."""
    b = _bits(bits)
    c, s, z = _canon(codes, scales, zeros, b)
    n = packed_size(shape, b)
    out = np.empty(n, np.uint8)
    _check(load().mc_pack_experts_host(ctypes.byref(shape), b.ctypes.data, _ptr_array(c, None),
                                       _ptr_array(s, None), _ptr_array(z, None), out.ctypes.data, n))
    return out


def unpack_experts_host(packed: np.ndarray, expert: int, mat: int, rows: int, cols: int, group: int):
    codes = np.empty((rows, cols), np.uint8)
    scale = np.empty((rows, cols // group), np.uint16)
    zero = np.empty((rows, cols // group), np.uint16)
    _check(load().mc_unpack_experts_host(packed.ctypes.data, packed.nbytes, expert, mat, codes.ctypes.data,
                                         scale.ctypes.data, zero.ctypes.data))
    return codes, scale.view(np.float16), zero.view(np.float16)


def pack_experts(shape: Shape, bits, codes, scales, zeros, device="cuda"):
    """Pack and upload; returns a uint8 device tensor (synchronous)."""
    import torch
    b = _bits(bits)
    c, s, z = _canon(codes, scales, zeros, b)
    n = packed_size(shape, b)
    dst = torch.empty(n, dtype=torch.uint8, device=device)
    _check(load().mc_pack_experts(ctypes.byref(shape), b.ctypes.data, _ptr_array(c, None), _ptr_array(s, None),
                                  _ptr_array(z, None), dst.data_ptr(), n, _stream()))
    return dst


def upload_packed(packed_host: np.ndarray, device="cuda"):
    """Copy an already packed host buffer to the device (uint8 tensor)."""
    import torch
    return torch.from_numpy(packed_host).to(device)


def unpack_experts(shape: Shape, bits, packed_dev, expert: int, mat: int, status=None):
    import torch
    rows, cols = (shape.F, shape.H) if mat < 2 else (shape.H, shape.F)
    dev = packed_dev.device
    codes = torch.empty((rows, cols), dtype=torch.uint8, device=dev)
    scale = torch.empty((rows, cols // shape.group), dtype=torch.float16, device=dev)
    zero = torch.empty((rows, cols // shape.group), dtype=torch.float16, device=dev)
    b = _bits(bits)
    _check(load().mc_unpack_experts(ctypes.byref(shape), b.ctypes.data, packed_dev.data_ptr(), expert, mat,
                                    codes.data_ptr(), scale.data_ptr(), zero.data_ptr(), _ptr(status), _stream()))
    return codes, scale, zero


def pack_verify(shape: Shape, bits, packed_dev) -> None:
    b = _bits(bits)
    _check(load().mc_pack_verify(ctypes.byref(shape), b.ctypes.data, packed_dev.data_ptr(), packed_dev.numel()))


# ------------------------------------------------------------------ routing --

def route(x, gate_w, shape: Shape, mu: float, protect=None):
    """Eq. 1 top-2 + Eq. 5 ODP + permutation.  protect: uint8 [T] token mask (0
    prunable, 2 dropped, other values protected) or None.  Returns a dict of
    device tensors."""
    import torch
    T = x.shape[0]
    dev = x.device
    out = {
        "idx": torch.empty((T, 2), dtype=torch.int32, device=dev),
        "w": torch.empty((T, 2), dtype=torch.float32, device=dev),
        "pruned": torch.empty(T, dtype=torch.uint8, device=dev),
        "offsets": torch.empty(shape.E + 1, dtype=torch.int32, device=dev),
        "perm": torch.empty(max(2 * T, 1), dtype=torch.int32, device=dev),
    }
    _check(load().mc_route(_ptr(x), _ptr(gate_w), T, ctypes.byref(shape), float(mu), _ptr(protect),
                           _ptr(out["idx"]), _ptr(out["w"]), _ptr(out["pruned"]), _ptr(out["offsets"]),
                           _ptr(out["perm"]), _stream()))
    return out


# -------------------------------------------------------------------- layer --

def workspace_size(shape: Shape, T: int) -> int:
    n = load().mc_moe_workspace_size(ctypes.byref(shape), int(T))
    if n == 0 and T > 0:
        raise MCError(ERR_INVALID_ARG, last_error())
    return n


def alloc_workspace(shape: Shape, T: int, device="cuda"):
    import torch
    n = workspace_size(shape, T)
    ws = torch.zeros(max(n, 256), dtype=torch.uint8, device=device)
    return ws


def moe_forward(x, gate_w, shape: Shape, bits, packed_dev, mu: float = 0.0, protect=None, y=None,
                workspace=None, routing: bool = False):
    """The whole layer.  x bf16 [T,H]; returns y bf16 [T,H] (and routing tensors)."""
    import torch
    T = x.shape[0]
    dev = x.device
    if y is None:
        y = torch.empty_like(x)
    if workspace is None:
        workspace = alloc_workspace(shape, T, dev)
    b = _bits(bits)
    idx = w = pr = None
    if routing:
        idx = torch.empty((T, 2), dtype=torch.int32, device=dev)
        w = torch.empty((T, 2), dtype=torch.float32, device=dev)
        pr = torch.empty(T, dtype=torch.uint8, device=dev)
    _check(load().mc_moe_forward(_ptr(x), _ptr(gate_w), T, ctypes.byref(shape), b.ctypes.data, _ptr(packed_dev),
                                 float(mu), _ptr(protect), _ptr(y), _ptr(workspace), workspace.numel(),
                                 _ptr(idx), _ptr(w), _ptr(pr), _stream()))
    if routing:
        return y, {"idx": idx, "w": w, "pruned": pr}
    return y


def moe_forward_static(x, gate_w, shape: Shape, bits, packed_dev, mu: float = 0.0, protect=None, y=None,
                       status=None):
    """mc_moe_forward_static: the layer with the library's fixed device scratch
    instead of a workspace.  `y` (bf16 [T,H]) and `status` (device int32, zeroed by
    the caller; None = the scratch's own status word) must already exist when the
    caller may not allocate."""
    import torch
    T = x.shape[0]
    if y is None:
        y = torch.empty_like(x)
    b = _bits(bits)
    _check(load().mc_moe_forward_static(_ptr(x), _ptr(gate_w), T, ctypes.byref(shape), b.ctypes.data,
                                        _ptr(packed_dev), float(mu), _ptr(protect), _ptr(y), _ptr(status),
                                        _stream()))
    return y


def stack_workspace(shape: Shape, T: int, device="cuda"):
    import torch
    n = load().mc_stack_workspace_size(ctypes.byref(shape), int(T))
    if n == 0:
        raise MCError(ERR_INVALID_ARG, last_error())
    return torch.zeros(n, dtype=torch.uint8, device=device)


class StackArgs:
    """Host-side argument arrays of mc_stack_forward, built once per stack so that
    repeated calls (or a captured graph) reuse the same host memory."""

    def __init__(self, gates, bits, packed, mus):
        self.layers = len(gates)
        self.gate_ptrs = (ctypes.c_void_p * self.layers)(*[g.data_ptr() for g in gates])
        self.packed_ptrs = (ctypes.c_void_p * self.layers)(*[p.data_ptr() for p in packed])
        self.bits = np.ascontiguousarray(np.concatenate([_bits(b) for b in bits]), dtype=np.int8)
        self.mus = np.ascontiguousarray(mus, dtype=np.float32)
        self._keep = (gates, packed)


def stack_forward(h, shape: Shape, args: StackArgs, gamma, workspace, protect=None, eps: float = 1e-5):
    """mc_stack_forward: h (bf16 [T,H], device) updated in place."""
    T = h.shape[0]
    _check(load().mc_stack_forward(_ptr(h), T, ctypes.byref(shape), args.layers,
                                   ctypes.cast(args.gate_ptrs, ctypes.c_void_p), args.bits.ctypes.data,
                                   ctypes.cast(args.packed_ptrs, ctypes.c_void_p), args.mus.ctypes.data,
                                   _ptr(protect), _ptr(gamma), float(eps), _ptr(workspace), workspace.numel(),
                                   _stream()))
    return h


def check_status(workspace) -> None:
    _check(load().mc_check_status(_ptr(workspace), _stream()))


def set_path(path: int) -> int:
    """Force the expert path of moe_forward (PATH_AUTO, PATH_GEMV, PATH_GEMM);
    returns the previous one."""
    r = load().mc_set_path(int(path))
    if r < 0:
        _check(r)
    return r


def set_debug(flags: int, timeout_ns: int = 0) -> None:
    load().mc_set_debug(int(flags), int(timeout_ns))


def rmsnorm(x, gamma, eps: float = 1e-5, out=None):
    import torch
    if out is None:
        out = torch.empty_like(x)
    T, H = x.shape
    _check(load().mc_rmsnorm(_ptr(x), _ptr(gamma), T, H, float(eps), _ptr(out), _stream()))
    return out


def add(a, b, out=None):
    import torch
    if out is None:
        out = torch.empty_like(a)
    _check(load().mc_add(_ptr(a), _ptr(b), a.numel(), _ptr(out), _stream()))
    return out


# -------------------------------------------------------------- profiling --

N_KERNELS = 11


def token_importance(t, attn, protect_frac: float = 0.02, importance=None, mask=None, with_mask: bool = True,
                     workspace=None):
    """Eq. 6 token importance of the tokens t (bf16 [L, H]) from the block's
    attention probabilities attn (fp32 [nh, L, L], query-major) and the protect
    mask of the top ceil(protect_frac * L) tokens.  Returns (importance, mask)."""
    import torch
    L, H = t.shape
    nh = attn.shape[0]
    assert attn.dtype == torch.float32 and tuple(attn.shape) == (nh, L, L) and attn.is_contiguous()
    if importance is None:
        importance = torch.empty(L, dtype=torch.float32, device=t.device)
    if with_mask and mask is None:
        mask = torch.empty(L, dtype=torch.uint8, device=t.device)
    if workspace is None:
        workspace = torch.empty(max(1, load().mc_token_importance_workspace_size(L)), dtype=torch.uint8,
                                device=t.device)
    _check(load().mc_token_importance(_ptr(t), _ptr(attn), L, H, nh, float(protect_frac), _ptr(importance),
                                      _ptr(mask) if with_mask else None, _ptr(workspace), workspace.numel(),
                                      _stream()))
    return importance, mask


def odp_threshold(w, mask=None, q: float = 0.5) -> float:
    """Eq. 5 threshold mu: the q-quantile of w1/w0 over the tokens with mask 0
    (w: routing weights [T, 2] from route(); host copies are taken)."""
    wh = np.ascontiguousarray(_host(w), dtype=np.float32)
    mh = None if mask is None else np.ascontiguousarray(_host(mask), dtype=np.uint8)
    mu = ctypes.c_float()
    _check(load().mc_odp_threshold_host(wh.ctypes.data, None if mh is None else mh.ctypes.data, wh.shape[0],
                                        float(q), ctypes.byref(mu)))
    return float(mu.value)


def expert_significance(idx, w, pruned, E: int):
    """Sec. 2.2.1: (phi, wact) per expert from routing outputs (host copies taken)."""
    i = np.ascontiguousarray(_host(idx), dtype=np.int32)
    ww = np.ascontiguousarray(_host(w), dtype=np.float32)
    p = None if pruned is None else np.ascontiguousarray(_host(pruned), dtype=np.uint8)
    phi, wact = np.empty(E), np.empty(E)
    _check(load().mc_expert_significance_host(i.ctypes.data, ww.ctypes.data, None if p is None else p.ctypes.data,
                                              i.shape[0], E, phi.ctypes.data, wact.ctypes.data))
    return phi, wact


def pmq_allocate(phi, wact, eps, bits_total: int, alpha: float = 1.0, beta: float = 1.0, gamma: float = 2.0):
    """Eq. 4 bit allocation (exact).  eps [E, 3].  Returns (bits int8 [E], objective)."""
    phi = np.ascontiguousarray(phi, dtype=np.float64)
    wact = np.ascontiguousarray(wact, dtype=np.float64)
    eps = np.ascontiguousarray(eps, dtype=np.float64)
    E = phi.shape[0]
    bits = np.empty(E, np.int8)
    obj = ctypes.c_double()
    _check(load().mc_pmq_allocate(phi.ctypes.data, wact.ctypes.data, eps.ctypes.data, E, int(bits_total),
                                  float(alpha), float(beta), float(gamma), bits.ctypes.data, ctypes.byref(obj)))
    return bits, float(obj.value)


def _host(a):
    try:
        import torch
        if isinstance(a, torch.Tensor):
            return a.detach().cpu().numpy()
    except ImportError:
        pass
    return np.asarray(a)


def profile_enable(on: bool = True) -> bool:
    return bool(load().mc_profile_enable(1 if on else 0))


def profile_select(names) -> None:
    """Record only the named kernels (None = all) while profiling is on."""
    if names is None:
        load().mc_profile_select(0xFFFFFFFF)
        return
    ids = [i for i in range(N_KERNELS) if load().mc_profile_name(i).decode() in set(names)]
    load().mc_profile_select(sum(1 << i for i in ids))


def profile_clear() -> None:
    """Drop every profiling record, including those of captured graphs."""
    _check(load().mc_profile_clear())


def profile_read() -> dict:
    """{kernel name: (total ms, launches)} since the last read."""
    ms = np.zeros(N_KERNELS, np.float64)
    cnt = np.zeros(N_KERNELS, np.int32)
    _check(load().mc_profile_read(ms.ctypes.data, cnt.ctypes.data, N_KERNELS))
    lib = load()
    return {lib.mc_profile_name(i).decode(): (float(ms[i]), int(cnt[i])) for i in range(N_KERNELS) if cnt[i]}


def selftest_umma(A, B, status=None, a_in_tmem=False):
    """D = A @ B.T through the tcgen05 path (A fp16 [128, K], B fp16 [N, K]);
    a_in_tmem: the A operand is staged in tensor memory instead of shared memory."""
    import torch
    D = torch.empty((A.shape[0], B.shape[0]), dtype=torch.float32, device=A.device)
    n = -B.shape[0] if a_in_tmem else B.shape[0]
    _check(load().mc_selftest_umma(_ptr(A), _ptr(B), _ptr(D), n, A.shape[1], _ptr(status), _stream()))
    return D


