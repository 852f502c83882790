"""ctypes binding of libember (include/ember.h), with the C names.

Argument marshalling only: every step runs in the CUDA kernels of the
library.  Pointers may be passed as integers or as torch tensors (their
data_ptr() is used); streams as integers, torch.cuda.Stream objects or None
(the current torch stream).  A non-OK status raises EmberError.  If the
compiled library is missing this module raises on import of the library
instead of falling back to anything else.
"""
import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libember.so")

EMBER_OK = 0
EMBER_ERR_INVALID_ARG = 1
EMBER_ERR_ALIGNMENT = 2
EMBER_ERR_DTYPE = 3
EMBER_ERR_WORKSPACE = 4
EMBER_ERR_CUDA = 5
EMBER_ERR_ID_OUT_OF_RANGE = 6
EMBER_ERR_TIMEOUT = 7
EMBER_ERR_UNSUPPORTED = 8

EMBER_F32 = 0
EMBER_BF16 = 1
EMBER_I32 = 0
EMBER_I64 = 1
EMBER_VARIANT_FULL = 0
EMBER_VARIANT_ROW = 1
EMBER_VARIANT_COL = 2

# Every function include/ember.h declares.
EXPORTS = (
    "ember_hparams_default", "ember_create", "ember_destroy", "ember_state_numel",
    "ember_workspace_bytes", "ember_bind_workspace", "ember_step_dense",
    "ember_step_sparse", "ember_get_device_status", "ember_status_string",
    "ember_abi_version", "ember_set_trace_events", "ember_sparse_unique",
    "ember_step_dense_noalloc", "ember_step_dense_from_host",
    "ember_lmhead_grad", "ember_step_lmhead",
    "ember_shard_rows", "ember_shard_scale_bytes", "ember_shard_exchange_bytes", "ember_shard_reduce",
    "ember_shard_pack", "ember_shard_update", "ember_column_panels", "ember_set_wait_limit_ns",
    "ember_dense_step_launches",
)


class ember_hparams(ctypes.Structure):
    _fields_ = [("beta2", ctypes.c_double), ("eps", ctypes.c_double),
                ("maximize", ctypes.c_int), ("bias_correction", ctypes.c_int),
                ("variant", ctypes.c_int)]


class EmberError(RuntimeError):
    def __init__(self, status, where=""):
        self.status = status
        super().__init__(f"{where}: {ember_status_string(status)} (status {status})")


_lib = None


def lib():
    """The loaded libember.so; raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(
                f"{LIB_PATH} is missing: build it with __graft_entry__.build() "
                "(there is no fallback implementation)")
        L = ctypes.CDLL(LIB_PATH)
        vp, i64, sz, st, flt, ip = (ctypes.c_void_p, ctypes.c_int64, ctypes.c_size_t,
                                    ctypes.c_int, ctypes.c_float, ctypes.c_int)
        hp = ctypes.POINTER(ember_hparams)
        sig = {
            "ember_hparams_default": (None, [hp]),
            "ember_create": (st, [i64, i64, hp, ip, ctypes.POINTER(vp)]),
            "ember_destroy": (None, [vp]),
            "ember_state_numel": (sz, [vp]),
            "ember_workspace_bytes": (sz, [vp, i64]),
            "ember_bind_workspace": (st, [vp, vp, sz, i64, vp]),
            "ember_step_dense": (st, [vp, vp, vp, vp, flt, i64, vp]),
            "ember_step_sparse": (st, [vp, vp, vp, ip, i64, vp, vp, flt, i64, vp]),
            "ember_get_device_status": (st, [vp, vp]),
            "ember_status_string": (ctypes.c_char_p, [st]),
            "ember_abi_version": (ip, []),
            "ember_set_trace_events": (st, [vp, ctypes.POINTER(vp), ip]),
            "ember_sparse_unique": (st, [vp, vp, ip, i64, vp, vp, vp, vp]),
            "ember_step_dense_noalloc": (st, [vp, vp, vp, vp, flt, i64, vp]),
            "ember_step_dense_from_host": (st, [vp, vp, vp, vp, vp, flt, i64, vp]),
            "ember_lmhead_grad": (st, [vp, vp, vp, i64, vp, vp]),
            "ember_step_lmhead": (st, [vp, vp, vp, vp, i64, vp, vp, flt, i64, vp]),
            "ember_shard_rows": (i64, [vp, ip, ip, ctypes.POINTER(i64)]),
            "ember_shard_scale_bytes": (sz, [vp]),
            "ember_shard_exchange_bytes": (sz, [vp]),
            "ember_shard_reduce": (st, [vp, ip, ip, vp, vp, vp, vp]),
            "ember_shard_pack": (st, [vp, ip, ip, vp, vp, vp]),
            "ember_shard_update": (st, [vp, ip, ip, vp, vp, vp, vp, vp, flt, i64, vp]),
            "ember_column_panels": (ip, [vp, ip]),
            "ember_dense_step_launches": (ip, [vp, ip]),
            "ember_set_wait_limit_ns": (st, [vp, ctypes.c_uint64]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def _addr(x):
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _stream(s):
    if s is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(s, int):
        return s
    return s.cuda_stream


def _check(status, where):
    if status != EMBER_OK:
        raise EmberError(status, where)


def ember_status_string(status):
    return lib().ember_status_string(status).decode()


def ember_abi_version():
    return lib().ember_abi_version()


def ember_column_panels(h, vector_path=True):
    """Column panels a step of this handle runs in (1 unless D is wider than
    one CTA's row)."""
    return lib().ember_column_panels(h, int(bool(vector_path)))


def ember_dense_step_launches(h, vector_path=True):
    """Kernel launches of one ember_step_dense of this handle (1 for a small table)."""
    return lib().ember_dense_step_launches(h, int(bool(vector_path)))


def ember_hparams_default():
    hp = ember_hparams()
    lib().ember_hparams_default(ctypes.byref(hp))
    return hp


def ember_create(V, D, hparams=None, wdtype=EMBER_BF16):
    """Returns the handle (an integer); raises EmberError on a bad argument."""
    out = ctypes.c_void_p()
    hp = ctypes.byref(hparams) if hparams is not None else None
    _check(lib().ember_create(V, D, hp, wdtype, ctypes.byref(out)), "ember_create")
    return out.value


def ember_destroy(h):
    lib().ember_destroy(h)


def ember_state_numel(h):
    return lib().ember_state_numel(h)


def ember_workspace_bytes(h, max_sparse_N=0):
    return lib().ember_workspace_bytes(h, max_sparse_N)


def ember_bind_workspace(h, workspace, nbytes, max_sparse_N=0, stream=None):
    _check(lib().ember_bind_workspace(h, _addr(workspace), nbytes, max_sparse_N, _stream(stream)),
           "ember_bind_workspace")


def ember_step_dense(h, W, G, state, lr, t, stream=None):
    _check(lib().ember_step_dense(h, _addr(W), _addr(G), _addr(state), lr, t, _stream(stream)),
           "ember_step_dense")


def ember_step_dense_noalloc(h, W, G, state, lr, t, stream=None):
    """The dense step with the library's own scratch array (no workspace)."""
    _check(lib().ember_step_dense_noalloc(h, _addr(W), _addr(G), _addr(state), lr, t,
                                          _stream(stream)), "ember_step_dense_noalloc")


def ember_step_dense_from_host(h, W, G_host, G_stage, state, lr, t, stream=None):
    """The dense step reading G from pinned host memory, staging it in G_stage."""
    _check(lib().ember_step_dense_from_host(h, _addr(W), _addr(G_host), _addr(G_stage), _addr(state),
                                            lr, t, _stream(stream)), "ember_step_dense_from_host")


def ember_lmhead_grad(h, dlogits, hidden, T, G, stream=None):
    """G = dlogits^T hidden on the tensor cores (dlogits T x V, hidden T x D, bf16)."""
    _check(lib().ember_lmhead_grad(h, _addr(dlogits), _addr(hidden), T, _addr(G), _stream(stream)),
           "ember_lmhead_grad")


def ember_step_lmhead(h, W, dlogits, hidden, T, G, state, lr, t, stream=None):
    """The dense step on G = dlogits^T hidden, formed (and written to G) here."""
    _check(lib().ember_step_lmhead(h, _addr(W), _addr(dlogits), _addr(hidden), T, _addr(G), _addr(state),
                                   lr, t, _stream(stream)), "ember_step_lmhead")


def ember_shard_rows(h, shard, nshards):
    """(row0, rows) that shard `shard` of `nshards` holds."""
    row0 = ctypes.c_int64(0)
    n = lib().ember_shard_rows(h, shard, nshards, ctypes.byref(row0))
    if n < 0:
        raise EmberError(EMBER_ERR_INVALID_ARG, "ember_shard_rows")
    return row0.value, n


def ember_shard_scale_bytes(h):
    """Bytes of a shard's exponent block (one uint8 per column, one for the r sums)."""
    return lib().ember_shard_scale_bytes(h)


def ember_shard_exchange_bytes(h):
    """Bytes of a shard's fixed-point block (one uint64 per column, one for the r sums)."""
    return lib().ember_shard_exchange_bytes(h)


def ember_shard_reduce(h, shard, nshards, G_shard, state, scales, stream=None):
    _check(lib().ember_shard_reduce(h, shard, nshards, _addr(G_shard), _addr(state), _addr(scales),
                                    _stream(stream)), "ember_shard_reduce")


def ember_shard_pack(h, shard, nshards, scales, sums, stream=None):
    _check(lib().ember_shard_pack(h, shard, nshards, _addr(scales), _addr(sums), _stream(stream)),
           "ember_shard_pack")


def ember_shard_update(h, shard, nshards, W_shard, G_shard, state, scales, sums, lr, t, stream=None):
    _check(lib().ember_shard_update(h, shard, nshards, _addr(W_shard), _addr(G_shard), _addr(state),
                                    _addr(scales), _addr(sums), lr, t, _stream(stream)), "ember_shard_update")


def ember_set_wait_limit_ns(h, ns):
    """Limit of the bounded waits inside this handle's kernels (0: the default, 2 s)."""
    _check(lib().ember_set_wait_limit_ns(h, int(ns)), "ember_set_wait_limit_ns")


def ember_step_sparse(h, W, ids, idtype, N, rows, state, lr, t, stream=None):
    _check(lib().ember_step_sparse(h, _addr(W), _addr(ids), idtype, N, _addr(rows), _addr(state),
                                   lr, t, _stream(stream)), "ember_step_sparse")


def ember_sparse_unique(h, ids, idtype, N, uniq, counts, n_unique, stream=None):
    _check(lib().ember_sparse_unique(h, _addr(ids), idtype, N, _addr(uniq), _addr(counts),
                                     _addr(n_unique), _stream(stream)), "ember_sparse_unique")


def ember_get_device_status(h, stream=None):
    """Synchronises the stream; returns (and clears) the sticky device status."""
    return lib().ember_get_device_status(h, _stream(stream))


def ember_set_trace_events(h, events):
    """events: torch.cuda.Event objects (created with enable_timing=True) or raw
    handles; [] stops tracing.  torch creates an event lazily, so each one is
    recorded once here to make sure it exists."""
    handles = []
    for ev in events:
        if isinstance(ev, int):
            handles.append(ev)
        else:
            ev.record()
            handles.append(ev.cuda_event)
    arr = (ctypes.c_void_p * max(len(handles), 1))(*handles)
    _check(lib().ember_set_trace_events(h, arr if handles else None, len(handles)),
           "ember_set_trace_events")


class Ember:
    """One token table's optimizer: the handle, its fp32 state (r then c) and
    its workspace, all device memory allocated through torch."""

    def __init__(self, V, D, wdtype="bf16", beta2=0.999, eps=1e-8, maximize=False,
                 bias_correction=True, variant="full", max_sparse_N=0, device="cuda"):
        import torch
        hp = ember_hparams(beta2=beta2, eps=eps, maximize=int(maximize),
                           bias_correction=int(bias_correction),
                           variant={"full": 0, "row": 1, "col": 2}[variant])
        self.V, self.D = V, D
        self.wdtype = {"bf16": EMBER_BF16, "f32": EMBER_F32}[wdtype]
        self.handle = ember_create(V, D, hp, self.wdtype)
        self.state = torch.zeros(ember_state_numel(self.handle), dtype=torch.float32, device=device)
        nbytes = ember_workspace_bytes(self.handle, max_sparse_N)
        self.workspace = torch.empty(nbytes, dtype=torch.uint8, device=device)
        self.max_sparse_N = max_sparse_N
        ember_bind_workspace(self.handle, self.workspace, nbytes, max_sparse_N)

    @property
    def r(self):
        return self.state[: self.V]

    @property
    def c(self):
        return self.state[self.V:]

    def step_dense(self, W, G, lr, t, stream=None):
        ember_step_dense(self.handle, W, G, self.state, lr, t, stream)

    def step_dense_from_host(self, W, G_host, G_stage, lr, t, stream=None):
        ember_step_dense_from_host(self.handle, W, G_host, G_stage, self.state, lr, t, stream)

    def lmhead_grad(self, dlogits, hidden, G, stream=None):
        """G (V x D fp32) = dlogits^T hidden; dlogits T x V and hidden T x D bf16."""
        ember_lmhead_grad(self.handle, dlogits, hidden, dlogits.shape[0], G, stream)

    def step_lmhead(self, W, dlogits, hidden, G, lr, t, stream=None):
        """One step of an LM head whose gradient dlogits^T hidden is formed into G."""
        ember_step_lmhead(self.handle, W, dlogits, hidden, dlogits.shape[0], G, self.state, lr, t, stream)

    # row-sharded dense step: this object is one shard's rank (its own
    # state and workspace); see include/ember.h for the protocol
    def shard_rows(self, shard, nshards):
        return ember_shard_rows(self.handle, shard, nshards)

    def shard_scale_bytes(self):
        return ember_shard_scale_bytes(self.handle)

    def shard_exchange_bytes(self):
        return ember_shard_exchange_bytes(self.handle)

    def shard_reduce(self, shard, nshards, G_shard, scales, stream=None):
        ember_shard_reduce(self.handle, shard, nshards, G_shard, self.state, scales, stream)

    def shard_pack(self, shard, nshards, scales, sums, stream=None):
        ember_shard_pack(self.handle, shard, nshards, scales, sums, stream)

    def shard_update(self, shard, nshards, W_shard, G_shard, scales, sums, lr, t, stream=None):
        ember_shard_update(self.handle, shard, nshards, W_shard, G_shard, self.state, scales, sums, lr, t,
                           stream)

    def set_wait_limit_ns(self, ns):
        ember_set_wait_limit_ns(self.handle, ns)

    def step_sparse(self, W, ids, rows, lr, t, stream=None):
        import torch
        idtype = EMBER_I64 if ids.dtype == torch.int64 else EMBER_I32
        ember_step_sparse(self.handle, W, ids, idtype, ids.numel(), rows, self.state, lr, t, stream)

    def unique(self, ids, stream=None):
        """(uniq, counts) of the valid ids, as int32 device tensors."""
        import torch
        idtype = EMBER_I64 if ids.dtype == torch.int64 else EMBER_I32
        n = ids.numel()
        uniq = torch.empty(max(n, 1), dtype=torch.int32, device=self.state.device)
        counts = torch.empty(max(n, 1), dtype=torch.int32, device=self.state.device)
        nu = torch.empty(1, dtype=torch.int32, device=self.state.device)
        ember_sparse_unique(self.handle, ids, idtype, n, uniq, counts, nu, stream)
        U = int(nu.item())
        return uniq[:U], counts[:U]

    def column_panels(self, vector_path=True):
        return ember_column_panels(self.handle, vector_path)

    def dense_step_launches(self, vector_path=True):
        return ember_dense_step_launches(self.handle, vector_path)

    def trace(self, events):
        ember_set_trace_events(self.handle, events)

    def device_status(self, stream=None):
        return ember_get_device_status(self.handle, stream)

    def close(self):
        if self.handle:
            ember_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
