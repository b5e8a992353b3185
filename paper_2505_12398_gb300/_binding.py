"""ctypes binding of libtv.so (C ABI in include/tv.h)."""

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))

TV_BF16 = 0
TV_FP32 = 1
# tv_create flags: which kernel path a handle uses ("auto" lets the library pick)
PATH_FLAGS = {"auto": 0, "three": 1, "cluster": 2, "persistent": 4}
# tv_create flags: the verification method ("token": the top-down token-level
# verifier the paper compares with; single-kernel paths only)
METHOD_FLAGS = {"traversal": 0, "token": 8}
TV_STATUS = {
    "BAD_TREE": 1,
    "BAD_TOKEN": 2,
    "DUP_SIBLING": 4,
    "ZERO_DRAFT": 8,
    "DEGENERATE": 16,
    "TIMEOUT": 32,
    "BAD_ROW": 64,
    "DRAFT_EXHAUSTED": 128,
}


class LibraryError(RuntimeError):
    """A call into libtv.so returned an error code."""

    def __init__(self, fn, code, lib):
        msg = lib.tv_strerror(code).decode() if lib is not None else "?"
        super().__init__(f"{fn} failed with code {code}: {msg}")
        self.code = code


def library_path():
    return os.path.join(HERE, "libtv.so")


_LIB = None

_P = ctypes.c_void_p
_I = ctypes.c_int
_F = ctypes.c_float

_SIGS = {
    "tv_create": (_I, [ctypes.POINTER(_P), _I, _I, _I, _I, _I, ctypes.c_uint]),
    "tv_verify_batch": (_I, [_P, _I, _I, _P, _P, _P, _P, _F, _P, _P, _P, _P, _P]),
    "tv_verify_batch_debug": (_I, [_P, _I, _I, _P, _P, _P, _P, _F, _P, _P, _P, _P, _P, _P, _P,
                                   _P]),
    "tv_verify_batch_host": (_I, [_P, _I, _I, _P, _P, _P, _P, _F, _P, _P, _P, _P, _P]),
    "tv_verify_batch_stats": (_I, [_P, _I, _I, _P, _P, _P, _P, _F, _P, _P, _P, _P, _P, _P, _P,
                                   _P]),
    "tv_lm_head": (_I, [_P, _I, _I, _P, _P, _F, _P, _P, _P]),
    "tv_draft_children": (_I, [_P, _I, _I, _P, _P, _P, _P, _P]),
    "tv_last_host_copy_bytes": (_I, [_P, _P, _P]),
    "tv_get_status": (_I, [_P, ctypes.POINTER(ctypes.c_uint32)]),
    "tv_debug_withhold_job": (_I, [_P, _I]),
    "tv_destroy": (_I, [_P]),
    "tv_set_phase_timing": (_I, [_P, _I]),
    "tv_last_phase_ms": (_I, [_P, ctypes.POINTER(ctypes.c_float)]),
    "tv_launch_shape": (_I, [_P, _I, _I, ctypes.POINTER(_I), ctypes.POINTER(_I),
                             ctypes.POINTER(_I), ctypes.POINTER(_I)]),
    "tv_verify_batch_noalloc": (_I, [_I, _I, _I, _I, _I, _P, _P, _P, _P, _F, _P, _P, _P, _P,
                                     _P]),
    "tv_strerror": (ctypes.c_char_p, [_I]),
    "tv_version": (_I, []),
}


def library():
    """Load libtv.so (raises if it has not been built: there is no fallback)."""
    global _LIB
    if _LIB is None:
        path = library_path()
        if not os.path.exists(path):
            raise ImportError(
                f"{path} is missing: build it with `python -m paper_2505_12398_gb300.build` "
                "(or __graft_entry__.build()); the verifier has no CPU implementation")
        lib = ctypes.CDLL(path)
        for name, (res, args) in _SIGS.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _LIB = lib
    return _LIB


def status_names(bits):
    return [k for k, v in TV_STATUS.items() if bits & v]


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr()) if t is not None else ctypes.c_void_p(0)


def _stream_ptr(stream):
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check_out(t, dtype, shape, device):
    """An output tensor the library writes: its dtype, shape, contiguity and
    device must be what the call's sizes say (the kernels trust them)."""
    if t.dtype != dtype or tuple(t.shape) != tuple(shape) or not t.is_contiguous() \
            or t.device != device:
        raise ValueError(f"output: expected a contiguous {dtype} {tuple(shape)} tensor on "
                         f"{device}, got {t.dtype} {tuple(t.shape)} on {t.device}")


class Verifier:
    """Owns a ``tv_handle`` (device workspace) for one device and size limits.

    All tensors passed to :meth:`verify` must be contiguous CUDA tensors on
    the handle's device with the dtypes and layouts of include/tv.h.
    """

    def __init__(self, vocab, max_nodes, max_batch, logit_dtype="bf16", device=0, path="auto",
                 method="traversal"):
        import torch
        self.lib = library()
        if logit_dtype in ("bf16", torch.bfloat16, TV_BF16):
            self.dtype_code, self.logit_dtype = TV_BF16, torch.bfloat16
        elif logit_dtype in ("fp32", torch.float32, TV_FP32):
            self.dtype_code, self.logit_dtype = TV_FP32, torch.float32
        else:
            raise ValueError(f"unsupported logit dtype {logit_dtype}")
        self.vocab, self.max_nodes, self.max_batch = vocab, max_nodes, max_batch
        self.device = torch.device("cuda", device) if isinstance(device, int) else torch.device(device)
        h = ctypes.c_void_p()
        if path not in PATH_FLAGS:
            raise ValueError(f"unknown path {path!r}; one of {sorted(PATH_FLAGS)}")
        if method not in METHOD_FLAGS:
            raise ValueError(f"unknown method {method!r}; one of {sorted(METHOD_FLAGS)}")
        self.method = method
        rc = self.lib.tv_create(ctypes.byref(h), self.device.index or 0, vocab, max_nodes,
                                max_batch, self.dtype_code,
                                PATH_FLAGS[path] | METHOD_FLAGS[method])
        if rc != 0:
            raise LibraryError("tv_create", rc, self.lib)
        self.handle = h

    def close(self):
        if getattr(self, "handle", None) is not None and self.handle.value:
            self.lib.tv_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _check(self, parents, tokens, logits, drafts, uniforms):
        import torch
        B, R = parents.shape
        N = R - 1
        V = self.vocab
        exp = [(parents, torch.int32, (B, R)), (tokens, torch.int32, (B, R)),
               (logits, self.logit_dtype, (B, R, V)), (drafts, torch.float32, (B, R, V)),
               (uniforms, torch.float32, (B, R + 1))]
        for t, dt, shape in exp:
            if t.dtype != dt or tuple(t.shape) != shape:
                raise ValueError(f"expected {dt} {shape}, got {t.dtype} {tuple(t.shape)}")
            if not t.is_contiguous():
                raise ValueError("tensors must be contiguous")
            if t.device != self.device:
                raise ValueError(f"tensor on {t.device}, handle on {self.device}")
        return B, N

    def verify(self, parents, tokens, logits, drafts, temperature, uniforms,
               out=None, stream=None, debug=False, margins=False):
        """Returns (path [B,N] int32, tau [B] int32, bonus [B] int32) as CUDA
        tensors, plus (node_p [B,N+1] f32, stats [B,5] int32) when ``debug``,
        plus margins [B,2] f32 (test, bonus) when ``margins`` too.
        Asynchronous on ``stream`` (default: torch's current stream)."""
        import torch
        B, N = self._check(parents, tokens, logits, drafts, uniforms)
        if out is None:
            path = torch.empty(B, N, dtype=torch.int32, device=self.device)
            tau = torch.empty(B, dtype=torch.int32, device=self.device)
            bonus = torch.empty(B, dtype=torch.int32, device=self.device)
        else:
            path, tau, bonus = out
            for t, shape in ((path, (B, N)), (tau, (B,)), (bonus, (B,))):
                _check_out(t, torch.int32, shape, self.device)
        sp = _stream_ptr(stream)
        if debug:
            node_p = torch.empty(B, N + 1, dtype=torch.float32, device=self.device)
            stats = torch.empty(B, 5, dtype=torch.int32, device=self.device)
            margin = torch.empty(B, 2, dtype=torch.float32, device=self.device)
            rc = self.lib.tv_verify_batch_debug(
                self.handle, B, N, _ptr(parents), _ptr(tokens), _ptr(logits), _ptr(drafts),
                float(temperature), _ptr(uniforms), _ptr(path), _ptr(tau), _ptr(bonus),
                _ptr(node_p), _ptr(stats), _ptr(margin), sp)
            if rc != 0:
                raise LibraryError("tv_verify_batch_debug", rc, self.lib)
            if margins:
                return path, tau, bonus, node_p, stats, margin
            return path, tau, bonus, node_p, stats
        rc = self.lib.tv_verify_batch(
            self.handle, B, N, _ptr(parents), _ptr(tokens), _ptr(logits), _ptr(drafts),
            float(temperature), _ptr(uniforms), _ptr(path), _ptr(tau), _ptr(bonus), sp)
        if rc != 0:
            raise LibraryError("tv_verify_batch", rc, self.lib)
        return path, tau, bonus

    def lm_head(self, hidden, weight, temperature, out=None, stream=None):
        """Logits [M, V] bf16 = hidden [M, K] x weight [V, K]^T on the tensor
        cores, and each row's normaliser [M, 2] fp32 (max, sum of
        2^((l - max) log2(e) / T)) of the stored logits (tv_lm_head).
        ``out`` = (logits, row_stats) to write into given tensors."""
        import torch
        M, K = hidden.shape
        for t, shape in ((hidden, (M, K)), (weight, (self.vocab, K))):
            if t.dtype != torch.bfloat16 or tuple(t.shape) != shape or not t.is_contiguous() \
                    or t.device != self.device:
                raise ValueError(f"expected a contiguous bf16 {shape} tensor on {self.device}")
        if out is None:
            logits = torch.empty(M, self.vocab, dtype=torch.bfloat16, device=self.device)
            row_stats = torch.empty(M, 2, dtype=torch.float32, device=self.device)
        else:
            logits, row_stats = out
            if logits.numel() != M * self.vocab or row_stats.numel() != 2 * M:
                raise ValueError("output: logits must hold M x V and row_stats M x 2 values")
            _check_out(logits, torch.bfloat16, logits.shape, self.device)
            _check_out(row_stats, torch.float32, row_stats.shape, self.device)
        rc = self.lib.tv_lm_head(self.handle, M, K, _ptr(hidden), _ptr(weight),
                                 float(temperature), _ptr(logits), _ptr(row_stats),
                                 _stream_ptr(stream))
        if rc != 0:
            raise LibraryError("tv_lm_head", rc, self.lib)
        return logits, row_stats

    def draft_children(self, parents, drafts, uniforms, out=None, stream=None):
        """Tokens [B, N+1] int32 of every node, drawn from its parent's draft
        row without its earlier siblings' tokens (Definition 1), node c with
        uniforms[:, c] (tv_draft_children).  parents [B, N+1] int32, drafts
        [B, N+1, V] fp32, uniforms [B, N+1] fp32, all on the handle's device."""
        import torch
        B, R = parents.shape
        for t, dt, shape in ((parents, torch.int32, (B, R)), (drafts, torch.float32, (B, R, self.vocab)),
                             (uniforms, torch.float32, (B, R))):
            if t.dtype != dt or tuple(t.shape) != shape or not t.is_contiguous() \
                    or t.device != self.device:
                raise ValueError(f"expected a contiguous {dt} {shape} tensor on {self.device}")
        tokens = torch.empty(B, R, dtype=torch.int32, device=self.device) if out is None else out
        _check_out(tokens, torch.int32, (B, R), self.device)
        rc = self.lib.tv_draft_children(self.handle, B, R - 1, _ptr(parents), _ptr(drafts),
                                        _ptr(uniforms), _ptr(tokens), _stream_ptr(stream))
        if rc != 0:
            raise LibraryError("tv_draft_children", rc, self.lib)
        return tokens

    def verify_stats(self, parents, tokens, logits, drafts, temperature, uniforms, row_stats,
                     out=None, stream=None, debug=False):
        """verify() with the rows' normalisers given ([B, N+1, 2] or [B*(N+1), 2]
        fp32, e.g. from lm_head) (tv_verify_batch_stats)."""
        import torch
        B, N = self._check(parents, tokens, logits, drafts, uniforms)
        if row_stats.dtype != torch.float32 or row_stats.numel() != 2 * B * (N + 1) or \
                not row_stats.is_contiguous() or row_stats.device != self.device:
            raise ValueError("row_stats must be a contiguous float32 [B*(N+1), 2] tensor "
                             "on the handle's device")
        if out is None:
            path = torch.empty(B, N, dtype=torch.int32, device=self.device)
            tau = torch.empty(B, dtype=torch.int32, device=self.device)
            bonus = torch.empty(B, dtype=torch.int32, device=self.device)
        else:
            path, tau, bonus = out
            for t, shape in ((path, (B, N)), (tau, (B,)), (bonus, (B,))):
                _check_out(t, torch.int32, shape, self.device)
        node_p = torch.empty(B, N + 1, dtype=torch.float32, device=self.device) if debug else None
        stats = torch.empty(B, 5, dtype=torch.int32, device=self.device) if debug else None
        rc = self.lib.tv_verify_batch_stats(
            self.handle, B, N, _ptr(parents), _ptr(tokens), _ptr(logits), _ptr(drafts),
            float(temperature), _ptr(uniforms), _ptr(row_stats), _ptr(path), _ptr(tau),
            _ptr(bonus), _ptr(node_p), _ptr(stats), _stream_ptr(stream))
        if rc != 0:
            raise LibraryError("tv_verify_batch_stats", rc, self.lib)
        return (path, tau, bonus, node_p, stats) if debug else (path, tau, bonus)

    def verify_host(self, parents, tokens, logits, drafts, temperature, uniforms,
                    out, stream=None):
        """Same verification from host (CPU, ideally pinned) tensors; copies in,
        verifies, copies the outputs into ``out`` = (path, tau, bonus) host
        tensors and synchronises."""
        B, R = parents.shape
        N = R - 1
        path, tau, bonus = out
        rc = self.lib.tv_verify_batch_host(
            self.handle, B, N, _ptr(parents), _ptr(tokens), _ptr(logits), _ptr(drafts),
            float(temperature), _ptr(uniforms), _ptr(path), _ptr(tau), _ptr(bonus),
            _stream_ptr(stream))
        if rc != 0:
            raise LibraryError("tv_verify_batch_host", rc, self.lib)
        return path, tau, bonus

    def last_host_copy_bytes(self):
        """(host-to-device, device-to-host) bytes of the last verify_host call
        (tv_last_host_copy_bytes)."""
        h2d, d2h = ctypes.c_uint64(), ctypes.c_uint64()
        rc = self.lib.tv_last_host_copy_bytes(self.handle, ctypes.byref(h2d), ctypes.byref(d2h))
        if rc != 0:
            raise LibraryError("tv_last_host_copy_bytes", rc, self.lib)
        return h2d.value, d2h.value

    def set_phase_timing(self, enable=True):
        rc = self.lib.tv_set_phase_timing(self.handle, 1 if enable else 0)
        if rc != 0:
            raise LibraryError("tv_set_phase_timing", rc, self.lib)

    def last_phase_ms(self):
        """Device milliseconds of (prep, row normalisers, traversal) of the
        last call made with phase timing on (waits for it)."""
        ms = (ctypes.c_float * 3)()
        rc = self.lib.tv_last_phase_ms(self.handle, ms)
        if rc != 0:
            raise LibraryError("tv_last_phase_ms", rc, self.lib)
        return [float(x) for x in ms]

    def launch_shape(self, B, N):
        """(path code, CTAs per tree, consumer warps per CTA, ring stages);
        path code 0 = three kernels, 1 = cluster per tree, 2 = persistent."""
        out = [ctypes.c_int() for _ in range(4)]
        rc = self.lib.tv_launch_shape(self.handle, B, N, *[ctypes.byref(o) for o in out])
        if rc != 0:
            raise LibraryError("tv_launch_shape", rc, self.lib)
        return tuple(o.value for o in out)

    def withhold_job(self, tree):
        """Test hook (tv_debug_withhold_job): the next persistent-kernel call
        never publishes tree ``tree``'s first job, so its waits run out."""
        rc = self.lib.tv_debug_withhold_job(self.handle, int(tree))
        if rc != 0:
            raise LibraryError("tv_debug_withhold_job", rc, self.lib)

    def status(self):
        """Synchronise and return (and clear) the TV_STATUS_* bits raised."""
        v = ctypes.c_uint32(0)
        rc = self.lib.tv_get_status(self.handle, ctypes.byref(v))
        if rc != 0:
            raise LibraryError("tv_get_status", rc, self.lib)
        return v.value
