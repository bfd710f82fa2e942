"""Python binding of libapc (include/apc.h): argument marshalling only.

Every step of the committed update and of the digest runs in the CUDA
kernels of ``libapc.so``; this module converts torch tensors (or raw device
pointers) into the C structures, calls the C ABI, and raises on a non-OK
status.  There is no CPU fallback: importing the binding without a built
library, or calling it without a CUDA device, raises.

Entry points mirror the C names:

* :func:`commit_step` -> ``apc_commit_step``: fused AdamW update of the fp32
  master shard and its moments from a bf16 gradient, the bf16 working copy,
  and the four state digests (p', m', v', w).
* :func:`digest` -> ``apc_digest``: the same digests of arbitrary buffers,
  read only (post-recovery verification).
* :func:`resolve_hparams` -> ``apc_resolve_hparams``: the step's binary32
  scalars (host only).
* :func:`upload` -> ``apc_upload``: host-to-device upload executed by a
  bounded number of CTAs, and :func:`set_reserved_sms` ->
  ``apc_set_reserved_sms``: SMs the persistent kernels leave free for it.

A table or buffer list that is used every step can be marshalled once with
:func:`prepare_table` / :func:`prepare_buffers` and passed in its place.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from typing import Iterable, Sequence

from . import _build

__all__ = ["TensorEntry", "TensorEntryBF16", "BufferEntry", "PreparedTable", "ApcError", "commit_step",
           "commit_step_bf16", "digest", "count_nonzero", "prepare_table", "prepare_buffers", "resolve_hparams",
           "Segment", "upload", "prepare_segments", "set_reserved_sms", "library", "lib_path", "F32", "BF16",
           "DEFAULT_HPARAMS"]

F32, BF16 = 0, 1
MASK64 = (1 << 64) - 1
DEFAULT_HPARAMS = dict(lr=3e-4, beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.1)


class _Tensor(ctypes.Structure):
    _fields_ = [("p", ctypes.c_void_p), ("m", ctypes.c_void_p), ("v", ctypes.c_void_p), ("g", ctypes.c_void_p),
                ("w", ctypes.c_void_p), ("n", ctypes.c_uint64), ("global_offset", ctypes.c_uint64)]


class _TensorBF16(ctypes.Structure):
    _fields_ = [("p", ctypes.c_void_p), ("m", ctypes.c_void_p), ("v", ctypes.c_void_p), ("g", ctypes.c_void_p),
                ("n", ctypes.c_uint64), ("global_offset", ctypes.c_uint64)]


class _Buffer(ctypes.Structure):
    _fields_ = [("data", ctypes.c_void_p), ("n", ctypes.c_uint64), ("global_offset", ctypes.c_uint64),
                ("dtype", ctypes.c_uint32), ("slot", ctypes.c_uint32)]


class _Segment(ctypes.Structure):
    _fields_ = [("dst", ctypes.c_void_p), ("src", ctypes.c_void_p), ("bytes", ctypes.c_uint64)]


class _HParams(ctypes.Structure):
    _fields_ = [("lr", ctypes.c_double), ("beta1", ctypes.c_double), ("beta2", ctypes.c_double),
                ("eps", ctypes.c_double), ("weight_decay", ctypes.c_double)]


class ApcError(RuntimeError):
    def __init__(self, status: int, detail: str):
        super().__init__("%s (%s)" % (detail, _lib_status_string(status)))
        self.status = status


_lib = None


def lib_path() -> str:
    return _build.LIB


def library():
    """Load libapc.so (building it first if it is missing or stale)."""
    global _lib
    if _lib is None:
        path = _build.build()
        lib = ctypes.CDLL(path)
        vp, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
        lib.apc_commit_step.argtypes = [vp, i32, vp, i64, vp, vp]
        lib.apc_commit_step.restype = ctypes.c_int
        lib.apc_commit_step_ex.argtypes = [vp, i32, vp, i64, ctypes.c_uint32, vp, vp]
        lib.apc_commit_step_ex.restype = ctypes.c_int
        lib.apc_commit_step_bf16.argtypes = [vp, i32, vp, i64, ctypes.c_uint32, vp, vp]
        lib.apc_commit_step_bf16.restype = ctypes.c_int
        lib.apc_count_nonzero.argtypes = [vp, i32, i32, vp, vp]
        lib.apc_count_nonzero.restype = ctypes.c_int
        lib.apc_digest.argtypes = [vp, i32, i32, vp, vp]
        lib.apc_digest.restype = ctypes.c_int
        lib.apc_resolve_hparams.argtypes = [vp, i64, vp]
        lib.apc_resolve_hparams.restype = ctypes.c_int
        lib.apc_status_string.argtypes = [ctypes.c_int]
        lib.apc_status_string.restype = ctypes.c_char_p
        lib.apc_last_error.argtypes = []
        lib.apc_last_error.restype = ctypes.c_char_p
        lib.apc_version.argtypes = []
        lib.apc_version.restype = ctypes.c_int32
        lib.apc_device_status.argtypes = []
        lib.apc_device_status.restype = ctypes.c_int
        lib.apc_selftest_wait_timeout.argtypes = [ctypes.c_uint64, vp]
        lib.apc_selftest_wait_timeout.restype = ctypes.c_int
        lib.apc_upload.argtypes = [vp, i32, i32, vp]
        lib.apc_upload.restype = ctypes.c_int
        lib.apc_set_reserved_sms.argtypes = [i32]
        lib.apc_set_reserved_sms.restype = ctypes.c_int
        _lib = lib
    return _lib


def _lib_status_string(status: int) -> str:
    return library().apc_status_string(status).decode()


def _check(status: int) -> None:
    if status != 0:
        raise ApcError(status, library().apc_last_error().decode() or "apc call failed")


def _hp(hp: dict | None) -> _HParams:
    hp = dict(DEFAULT_HPARAMS, **(hp or {}))
    return _HParams(hp["lr"], hp["beta1"], hp["beta2"], hp["eps"], hp["weight_decay"])


def _ptr(x, itemsize: int | None = None) -> int:
    """Device address of a torch tensor (checked: on the current CUDA device,
    contiguous, element size) or a raw integer pointer.  The library launches
    on the calling thread's current device, so a tensor of another device is
    refused here rather than dereferenced there."""
    if x is None:
        return 0
    if isinstance(x, int):
        return x
    if not x.is_cuda:
        raise ValueError("tensor is not on a CUDA device")
    import torch
    cur = torch.cuda.current_device()
    if x.device.index != cur:
        raise ValueError("tensor is on cuda:%s but the current device is cuda:%d (use torch.cuda.device(...))"
                         % (x.device.index, cur))
    if not x.is_contiguous():
        raise ValueError("tensor is not contiguous")
    if itemsize is not None and x.element_size() != itemsize:
        raise ValueError("expected %d-byte elements, got %s" % (itemsize, x.dtype))
    return x.data_ptr()


def _stream(stream) -> int:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


@dataclass
class TensorEntry:
    """One chunk-table entry: fp32 p, m, v (updated in place), bf16 g (read),
    bf16 w (written), n elements whose first has index ``global_offset`` in
    the flat model.  Fields are torch tensors or raw device pointers."""
    p: object
    m: object
    v: object
    g: object
    w: object
    global_offset: int = 0
    n: int | None = None

    def count(self) -> int:
        if self.n is not None:
            return int(self.n)
        return int(self.p.numel())


@dataclass
class TensorEntryBF16:
    """One entry of a bf16-state chunk table: bf16 p, m, v (updated in
    place) and bf16 g (read), n elements at ``global_offset``."""
    p: object
    m: object
    v: object
    g: object
    global_offset: int = 0
    n: int | None = None

    def count(self) -> int:
        if self.n is not None:
            return int(self.n)
        return int(self.p.numel())


@dataclass
class BufferEntry:
    """One digest buffer: ``data`` (torch tensor or pointer) of ``dtype``
    (F32 or BF16), n elements at ``global_offset``, summed into ``slot``."""
    data: object
    slot: int
    global_offset: int = 0
    dtype: int | None = None
    n: int | None = None


def _out(out, nslots: int, like):
    if out is not None:
        return out
    import torch
    dev = like.device if hasattr(like, "device") else torch.device("cuda", torch.cuda.current_device())
    return torch.empty(nslots, dtype=torch.int64, device=dev)


COMMIT_ZERO_GRAD = 1


class PreparedTable:
    """A chunk table or buffer list marshalled once into its C array, for
    repeated calls over the same buffers (a training job's table does not
    change between steps).  It keeps references to the tensors it points
    into, so their memory stays allocated while it lives."""

    def __init__(self, kind: str, arr, count: int, first, keep: list):
        self.kind, self.arr, self.count, self.first, self._keep = kind, arr, count, first, keep

    def __len__(self) -> int:
        return self.count


def _commit_array(table, kind: str):
    if isinstance(table, PreparedTable):
        if table.kind != kind:
            raise ValueError("prepared table is a %s table, expected %s" % (table.kind, kind))
        return table.arr, table.count, table.first
    table = list(table)
    if kind == "f32":
        arr = (_Tensor * max(1, len(table)))()
        fields = (("p", 4), ("m", 4), ("v", 4), ("g", 2), ("w", 2))
    else:
        arr = (_TensorBF16 * max(1, len(table)))()
        fields = (("p", 2), ("m", 2), ("v", 2), ("g", 2))
    first = None
    for i, t in enumerate(table):
        n = t.count()
        ptrs = []
        for name, size in fields:
            buf = getattr(t, name)
            if not isinstance(buf, int) and buf is not None and buf.numel() < n:
                raise ValueError("table[%d].%s has %d < %d elements" % (i, name, buf.numel(), n))
            ptrs.append(_ptr(buf, size))
        arr[i] = (_Tensor if kind == "f32" else _TensorBF16)(*ptrs, n, int(t.global_offset) & MASK64)
        if first is None and not isinstance(t.p, int):
            first = t.p
    return arr, len(table), first


def prepare_table(table: Sequence[TensorEntry] | Sequence[TensorEntryBF16]) -> PreparedTable:
    """Marshal a chunk table once (fp32-state entries for :func:`commit_step`,
    bf16-state entries for :func:`commit_step_bf16`)."""
    table = list(table)
    kind = "bf16" if table and isinstance(table[0], TensorEntryBF16) else "f32"
    arr, n, first = _commit_array(table, kind)
    return PreparedTable(kind, arr, n, first, table)


def commit_step(table: Sequence[TensorEntry] | PreparedTable, step: int, hparams: dict | None = None, stream=None,
                out=None, zero_grad: bool = False):
    """Enqueue the committed AdamW step + digest over ``table`` on ``stream``
    (``apc_commit_step``, or ``apc_commit_step_ex`` with
    APC_COMMIT_ZERO_GRAD when ``zero_grad``: the gradients are also zeroed).
    ``table`` is a list of :class:`TensorEntry` or a :class:`PreparedTable`.

    Returns the device int64[4] tensor that receives {D_p', D_m', D_v', D_w}
    (bit patterns of the unsigned digests; see :func:`digests_to_host`)."""
    arr, n, first = _commit_array(table, "f32")
    out = _out(out, 4, first)
    hp = _hp(hparams)
    if zero_grad:
        _check(library().apc_commit_step_ex(ctypes.addressof(arr), n, ctypes.addressof(hp), int(step),
                                            COMMIT_ZERO_GRAD, ctypes.c_void_p(_stream(stream)),
                                            ctypes.c_void_p(_ptr(out, 8))))
    else:
        _check(library().apc_commit_step(ctypes.addressof(arr), n, ctypes.addressof(hp), int(step),
                                         ctypes.c_void_p(_stream(stream)), ctypes.c_void_p(_ptr(out, 8))))
    return out


def commit_step_bf16(table: Sequence[TensorEntryBF16] | PreparedTable, step: int, hparams: dict | None = None,
                     stream=None, out=None, zero_grad: bool = False):
    """Enqueue the bf16-state committed step (``apc_commit_step_bf16``).
    Returns the device int64[3] tensor of {D_p', D_m', D_v'}."""
    arr, n, first = _commit_array(table, "bf16")
    out = _out(out, 3, first)
    hp = _hp(hparams)
    _check(library().apc_commit_step_bf16(ctypes.addressof(arr), n, ctypes.addressof(hp), int(step),
                                          COMMIT_ZERO_GRAD if zero_grad else 0, ctypes.c_void_p(_stream(stream)),
                                          ctypes.c_void_p(_ptr(out, 8))))
    return out


def _buffers(buffers):
    if isinstance(buffers, PreparedTable):
        if buffers.kind != "buffers":
            raise ValueError("prepared table is a %s table, expected a buffer list" % buffers.kind)
        return buffers.arr, buffers.count, buffers.first
    buffers = list(buffers)
    arr = (_Buffer * max(1, len(buffers)))()
    first = None
    for i, b in enumerate(buffers):
        dt = b.dtype
        if dt is None:
            if isinstance(b.data, int):
                raise ValueError("buffers[%d]: dtype is required for a raw pointer" % i)
            dt = F32 if b.data.element_size() == 4 else BF16
        n = b.n if b.n is not None else b.data.numel()
        arr[i] = _Buffer(_ptr(b.data, 4 if dt == F32 else 2), int(n), int(b.global_offset) & MASK64, dt,
                         int(b.slot))
        if first is None and not isinstance(b.data, int):
            first = b.data
    return arr, len(buffers), first


def prepare_buffers(buffers: Iterable[BufferEntry]) -> PreparedTable:
    """Marshal a buffer list once for :func:`digest` and :func:`count_nonzero`."""
    buffers = list(buffers)
    arr, n, first = _buffers(buffers)
    return PreparedTable("buffers", arr, n, first, buffers)


def digest(buffers: Iterable[BufferEntry] | PreparedTable, num_slots: int = 4, stream=None, out=None):
    """Enqueue the read-only digest of ``buffers`` (a list of
    :class:`BufferEntry` or a :class:`PreparedTable`) into ``num_slots``
    slots (``apc_digest``).  Returns the device int64[num_slots] output
    tensor."""
    arr, n, first = _buffers(buffers)
    out = _out(out, num_slots, first)
    _check(library().apc_digest(ctypes.addressof(arr), n, int(num_slots), ctypes.c_void_p(_stream(stream)),
                                ctypes.c_void_p(_ptr(out, 8))))
    return out


def count_nonzero(buffers: Iterable[BufferEntry] | PreparedTable, num_slots: int = 1, stream=None, out=None):
    """Enqueue the quiescence guard (``apc_count_nonzero``): per-slot counts
    of nonzero words.  Returns the device int64[num_slots] output tensor."""
    arr, n, first = _buffers(buffers)
    out = _out(out, num_slots, first)
    _check(library().apc_count_nonzero(ctypes.addressof(arr), n, int(num_slots), ctypes.c_void_p(_stream(stream)),
                                       ctypes.c_void_p(_ptr(out, 8))))
    return out


@dataclass
class Segment:
    """One upload segment: ``bytes`` bytes from ``src`` (a page-locked CPU
    tensor, a CUDA tensor, or a raw pointer the device can read) to ``dst``
    (a CUDA tensor or raw device pointer).  ``bytes`` defaults to dst's size."""
    dst: object
    src: object
    bytes: int | None = None


def _addr(x) -> int:
    if isinstance(x, int):
        return x
    if not x.is_contiguous():
        raise ValueError("tensor is not contiguous")
    return x.data_ptr()


def _segments(segments):
    if isinstance(segments, PreparedTable):
        if segments.kind != "segments":
            raise ValueError("prepared table is a %s table, expected a segment list" % segments.kind)
        return segments.arr, segments.count
    segments = list(segments)
    arr = (_Segment * max(1, len(segments)))()
    for i, g in enumerate(segments):
        n = g.bytes
        if n is None:
            n = g.dst.numel() * g.dst.element_size()
        for name, t in (("dst", g.dst), ("src", g.src)):
            if not isinstance(t, int) and t.numel() * t.element_size() < n:
                raise ValueError("segments[%d].%s holds fewer than %d bytes" % (i, name, n))
        if not isinstance(g.dst, int) and not g.dst.is_cuda:
            raise ValueError("segments[%d].dst is not a CUDA tensor" % i)
        arr[i] = _Segment(_addr(g.dst), _addr(g.src), int(n))
    return arr, len(segments)


def prepare_segments(segments: Iterable[Segment]) -> PreparedTable:
    """Marshal an upload segment list once for :func:`upload`."""
    segments = list(segments)
    arr, n = _segments(segments)
    return PreparedTable("segments", arr, n, None, segments)


def upload(segments: Iterable[Segment] | PreparedTable, max_ctas: int = 0, stream=None) -> None:
    """Enqueue the SM-driven host-to-device upload of ``segments`` on at
    most ``max_ctas`` CTAs (``apc_upload``; 0 = one per SM)."""
    arr, n = _segments(segments)
    _check(library().apc_upload(ctypes.addressof(arr), n, int(max_ctas), ctypes.c_void_p(_stream(stream))))


def set_reserved_sms(n: int) -> None:
    """Leave ``n`` SMs free of the library's persistent kernels
    (``apc_set_reserved_sms``; 0 restores the default)."""
    _check(library().apc_set_reserved_sms(int(n)))


def digests_to_host(out) -> list[int]:
    """Copy a digest tensor to the host as unsigned 64-bit Python ints."""
    return [int(x) & MASK64 for x in out.cpu().tolist()]


def resolve_hparams(hparams: dict | None, step: int) -> list[float]:
    """The eight binary32 scalars of step ``step`` (host only)."""
    hp = _hp(hparams)
    out = (ctypes.c_float * 8)()
    _check(library().apc_resolve_hparams(ctypes.addressof(hp), int(step), ctypes.addressof(out)))
    return list(out)


def device_status() -> int:
    """Synchronize the device and return (and clear) the kernels' device
    status: 0, or 5 (APC_ETIMEOUT) if a bounded wait inside a kernel gave up."""
    return int(library().apc_device_status())


def selftest_wait_timeout(limit_ns: int, stream=None) -> None:
    """Launch the bounded-wait self-test: a wait that nothing completes gives
    up after ``limit_ns`` and records APC_ETIMEOUT for :func:`device_status`."""
    _check(library().apc_selftest_wait_timeout(int(limit_ns), ctypes.c_void_p(_stream(stream))))


def state_buffers(p, m, v, w, global_offset: int = 0) -> list[BufferEntry]:
    """The four digest buffers of one tensor in commit_step's slot order."""
    return [BufferEntry(p, 0, global_offset, F32), BufferEntry(m, 1, global_offset, F32),
            BufferEntry(v, 2, global_offset, F32), BufferEntry(w, 3, global_offset, BF16)]


def state_buffers_bf16(p, m, v, global_offset: int = 0) -> list[BufferEntry]:
    """The three digest buffers of one bf16-state tensor in
    commit_step_bf16's slot order."""
    return [BufferEntry(p, 0, global_offset, BF16), BufferEntry(m, 1, global_offset, BF16),
            BufferEntry(v, 2, global_offset, BF16)]


__all__ += ["digests_to_host", "state_buffers", "device_status", "selftest_wait_timeout", "count_nonzero",
            "COMMIT_ZERO_GRAD", "TensorEntryBF16", "commit_step_bf16", "state_buffers_bf16"]
