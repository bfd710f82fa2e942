"""The C ABI without a GPU: the library builds and loads, exports every
function that include/apc.h declares, resolves the step scalars exactly as
the oracle does, and rejects bad arguments before touching the device."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle
import paper_2609_18178_gb300 as apc

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "apc.h")
M64 = (1 << 64) - 1


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^[A-Za-z_][\w\s\*]*?\b(apc_\w+)\s*\(", src, flags=re.M)))


def test_exports_every_declared_function():
    names = declared_functions()
    assert set(names) >= {"apc_commit_step", "apc_digest", "apc_resolve_hparams", "apc_status_string",
                          "apc_last_error", "apc_version", "apc_upload", "apc_set_reserved_sms"}
    lib = ctypes.CDLL(apc.lib_path() if os.path.exists(apc.lib_path()) else apc._build.build())
    for n in names:
        assert hasattr(lib, n), n
    assert apc.library().apc_version() == 3


def test_status_strings():
    lib = apc.library()
    for s in range(6):
        assert lib.apc_status_string(s).startswith(b"APC_")
    assert b"unknown" in lib.apc_status_string(99)


@pytest.mark.parametrize("hp", [oracle.DEFAULT_HP, dict(lr=1e-3, beta1=0.0, beta2=0.999, eps=1e-6, weight_decay=0.0),
                                dict(lr=0.0, beta1=0.5, beta2=0.5, eps=1e-12, weight_decay=0.3)])
@pytest.mark.parametrize("step", [1, 2, 3, 5, 10, 18, 1000, 1 << 40])
def test_resolve_hparams_matches_oracle_bitwise(hp, step):
    got = np.array(apc.resolve_hparams(hp, step), dtype=np.float32)
    want = oracle.resolve_hparams(hp, step)
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))


class _T(ctypes.Structure):
    _fields_ = [("p", ctypes.c_void_p), ("m", ctypes.c_void_p), ("v", ctypes.c_void_p), ("g", ctypes.c_void_p),
                ("w", ctypes.c_void_p), ("n", ctypes.c_uint64), ("global_offset", ctypes.c_uint64)]


class _B(ctypes.Structure):
    _fields_ = [("data", ctypes.c_void_p), ("n", ctypes.c_uint64), ("global_offset", ctypes.c_uint64),
                ("dtype", ctypes.c_uint32), ("slot", ctypes.c_uint32)]


def _hp(**kw):
    h = dict(oracle.DEFAULT_HP, **kw)
    return apc._HParams(h["lr"], h["beta1"], h["beta2"], h["eps"], h["weight_decay"])


def commit(table, step=1, hp=None, out=0x10000):
    lib = apc.library()
    arr = (_T * max(1, len(table)))(*table)
    h = hp if hp is not None else _hp()
    return lib.apc_commit_step(ctypes.addressof(arr) if table is not None else None, len(table or []),
                               ctypes.addressof(h), step, None, ctypes.c_void_p(out))


# fake device addresses: never dereferenced, the calls fail validation first
BASE = 0x7F0000000000


def fake(n, p=0, m=1 << 30, v=2 << 30, g=3 << 30, w=4 << 30, goff=0):
    return _T(BASE + p, BASE + m, BASE + v, BASE + g, BASE + w, n, goff)


def test_rejects_bad_scalars_and_step():
    assert commit([fake(8)], step=0) == 1
    assert commit([fake(8)], hp=_hp(beta1=1.0)) == 1
    assert commit([fake(8)], hp=_hp(eps=-1.0)) == 1
    assert commit([fake(8)], hp=_hp(lr=float("inf"))) == 1


def test_rejects_null_and_counts():
    lib = apc.library()
    h = _hp()
    assert lib.apc_commit_step(None, 1, ctypes.addressof(h), 1, None, ctypes.c_void_p(0x10000)) == 1
    assert lib.apc_commit_step(None, -1, ctypes.addressof(h), 1, None, ctypes.c_void_p(0x10000)) == 1
    assert commit([fake(8)], out=0) == 1
    assert commit([fake(8, p=0)], out=0x10004) == 2           # digests need 8-byte alignment
    t = fake(8)
    t.g = None
    assert commit([t]) == 1
    assert b"null" in apc.library().apc_last_error()


def test_rejects_misalignment_and_range():
    assert commit([fake(8, p=2)]) == 2
    assert commit([fake(8, g=1)]) == 2
    assert commit([fake(8, w=3)]) == 2
    assert commit([fake(100, goff=M64 - 50)]) == 3


def test_rejects_overlapping_outputs():
    assert commit([fake(100, p=0, m=200)]) == 1                # p [0,400) meets m [200, 600)
    assert commit([fake(100, g=0)]) == 1                       # gradient inside the p range
    a = fake(100)
    b = fake(100, p=8, m=(1 << 30) + 8000, v=(2 << 30) + 8000, g=(3 << 30) + 8000, w=(4 << 30) + 8000)
    assert commit([a, b]) == 1                                 # p ranges of two entries overlap


def test_digest_argument_checks():
    lib = apc.library()

    def dig(bufs, slots, out=0x10000):
        arr = (_B * max(1, len(bufs)))(*bufs)
        return lib.apc_digest(ctypes.addressof(arr), len(bufs), slots, None, ctypes.c_void_p(out))

    good = _B(BASE, 16, 0, 0, 0)
    assert dig([good], 0) == 1
    assert dig([good], 9) == 1
    assert dig([_B(BASE, 16, 0, 2, 0)], 4) == 1               # unknown dtype
    assert dig([_B(BASE, 16, 0, 0, 4)], 4) == 1               # slot >= num_slots
    assert dig([_B(BASE + 2, 16, 0, 0, 0)], 4) == 2           # fp32 needs 4-byte alignment
    assert dig([_B(BASE + 1, 16, 0, 1, 0)], 4) == 2           # bf16 needs 2-byte alignment
    assert dig([_B(None, 16, 0, 0, 0)], 4) == 1
    assert dig([_B(BASE, 100, M64 - 10, 0, 0)], 4) == 3
    assert dig([good], 4, out=0) == 1


def test_selftest_limit_checked():
    lib = apc.library()
    assert lib.apc_selftest_wait_timeout(0, None) == 1
    assert lib.apc_selftest_wait_timeout(10**11, None) == 1


def _no_device():
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("these calls pass validation with fake addresses: only without a device")


def test_valid_call_without_device_reports_cuda_error():
    """A call that passes argument validation next asks the runtime which
    device owns each pointer; without a device that query fails and the call
    returns APC_ECUDA before anything is enqueued."""
    _no_device()
    assert commit([fake(8)]) == 4
    assert apc.library().apc_last_error().startswith((b"cudaGetDevice", b"cudaPointerGetAttributes"))


def test_outputs_overlapping_inputs_are_rejected():
    """out_digests (commit) and the output of apc_digest / apc_count_nonzero
    are written ranges: meeting any buffer of the call is APC_EINVAL, found
    on the host before any CUDA call."""
    lib = apc.library()
    assert commit([fake(100)], out=BASE + 64) == 1                       # inside p
    assert commit([fake(100)], out=BASE + (3 << 30) + 8) == 1            # inside the gradient
    assert commit([fake(100)], out=BASE + (4 << 30) + 192) == 1          # inside w (200 bytes)
    assert b"out_digests" in lib.apc_last_error()

    def dig(fn, bufs, slots, out):
        arr = (_B * max(1, len(bufs)))(*bufs)
        return fn(ctypes.addressof(arr), len(bufs), slots, None, ctypes.c_void_p(out))

    for fn in (lib.apc_digest, lib.apc_count_nonzero):
        assert dig(fn, [_B(BASE, 16, 0, 0, 0)], 1, BASE + 56) == 1       # last 8 bytes of 64
        assert dig(fn, [_B(BASE, 16, 0, 0, 0)], 4, BASE - 24) == 1      # slots 3 meets the buffer
        assert b"overlaps" in lib.apc_last_error()


def test_binding_refuses_a_tensor_of_another_device(monkeypatch):
    """The binding passes only tensors of the current device to the library."""
    torch = pytest.importorskip("torch")

    class Fake:
        is_cuda = True
        device = torch.device("cuda", 1)

        def is_contiguous(self):
            return True

        def element_size(self):
            return 4

        def data_ptr(self):
            return BASE

    monkeypatch.setattr(torch.cuda, "current_device", lambda: 0)
    with pytest.raises(ValueError, match="current device"):
        apc._ptr(Fake(), 4)


def test_shared_gradient_is_not_an_overlap():
    """Two entries may read the same gradient range; only written ranges must
    be disjoint.  Without a device the call gets past validation and stops
    at the first CUDA call."""
    _no_device()
    a = fake(100)
    c = fake(100, p=4000, m=(1 << 30) + 4000, v=(2 << 30) + 4000, g=(3 << 30), w=(4 << 30) + 4000)
    assert commit([a, c]) == 4


def test_commit_ex_flags_and_zero_grad_overlap():
    lib = apc.library()
    h = _hp()

    def ex(table, flags):
        arr = (_T * max(1, len(table)))(*table)
        return lib.apc_commit_step_ex(ctypes.addressof(arr), len(table), ctypes.addressof(h), 1, flags, None,
                                      ctypes.c_void_p(0x10000))

    assert ex([fake(8)], 2) == 1                                # unknown flag bit
    a = fake(100)
    c = fake(100, p=4000, m=(1 << 30) + 4000, v=(2 << 30) + 4000, g=(3 << 30), w=(4 << 30) + 4000)
    assert ex([a, c], 1) == 1                                   # zeroing makes a shared gradient a written overlap


def test_count_nonzero_argument_checks():
    lib = apc.library()

    def cnt(bufs, slots, out=0x10000):
        arr = (_B * max(1, len(bufs)))(*bufs)
        return lib.apc_count_nonzero(ctypes.addressof(arr), len(bufs), slots, None, ctypes.c_void_p(out))

    assert cnt([_B(BASE, 16, 0, 0, 0)], 0) == 1
    assert cnt([_B(BASE, 16, 0, 3, 0)], 1) == 1
    assert cnt([_B(BASE + 1, 16, 0, 1, 0)], 1) == 2
    assert cnt([_B(BASE, 16, 0, 0, 0)], 1, out=0x10001) == 2


def test_prepared_table_marshals_like_the_list():
    """prepare_table / prepare_buffers build the same C arrays as the list
    forms, keep their kind, and the library validates them the same way."""
    e = [apc.TensorEntry(BASE, BASE + (1 << 30), BASE + (2 << 30), BASE + (3 << 30), BASE + (4 << 30), 7, n=100),
         apc.TensorEntry(BASE + 400, BASE + (1 << 30) + 400, BASE + (2 << 30) + 400, BASE + (3 << 30) + 200,
                         BASE + (4 << 30) + 200, 107, n=5)]
    t = apc.prepare_table(e)
    arr, n, _ = apc._commit_array(e, "f32")
    assert t.kind == "f32" and len(t) == n == 2 and bytes(t.arr) == bytes(arr)
    bad = apc.prepare_table([apc.TensorEntry(BASE + 2, BASE + (1 << 30), BASE + (2 << 30), BASE + (3 << 30),
                                             BASE + (4 << 30), 0, n=8)])
    with pytest.raises(apc.ApcError) as ei:
        apc.commit_step(bad, 1, stream=0, out=0x10000)
    assert ei.value.status == 2
    with pytest.raises(ValueError):
        apc.commit_step_bf16(t, 1, stream=0, out=0x10000)
    with pytest.raises(ValueError):
        apc.digest(t, 4, stream=0, out=0x10000)
    b = apc.prepare_buffers([apc.BufferEntry(BASE + 2, 0, 0, apc.F32, n=16)])
    assert b.kind == "buffers" and len(b) == 1
    with pytest.raises(apc.ApcError) as ei:
        apc.digest(b, 4, stream=0, out=0x10000)
    assert ei.value.status == 2
    with pytest.raises(ValueError):
        apc.commit_step(b, 1, stream=0, out=0x10000)


class _S(ctypes.Structure):
    _fields_ = [("dst", ctypes.c_void_p), ("src", ctypes.c_void_p), ("bytes", ctypes.c_uint64)]


def test_upload_and_reserve_argument_checks():
    lib = apc.library()

    def up(segs, ctas=0):
        arr = (_S * max(1, len(segs)))(*segs)
        return lib.apc_upload(ctypes.addressof(arr), len(segs), ctas, None)

    assert lib.apc_upload(None, 1, 0, None) == 1
    assert lib.apc_upload(None, 0, 0, None) == 0                # nothing to do
    assert up([_S(BASE, BASE + (1 << 30), 64)], ctas=-1) == 1
    assert up([_S(BASE, BASE + (1 << 30), 64)], ctas=5000) == 1
    assert up([_S(None, BASE, 64)]) == 1
    assert up([_S(BASE, None, 64)]) == 1
    assert up([_S(M64 - 10, BASE, 100)]) == 3                  # address + bytes overflows
    assert up([_S(None, None, 0), _S(BASE, BASE, 0)]) == 0     # empty segments are skipped
    assert lib.apc_set_reserved_sms(-1) == 1
    assert lib.apc_set_reserved_sms(1025) == 1
    assert lib.apc_set_reserved_sms(0) == 0


def test_last_error_is_per_thread():
    """Threads that fail validation in different ways at the same time each
    read back their own error detail (apc_last_error is thread-local)."""
    import threading
    lib = apc.library()
    cases = [
        (lambda: commit([fake(8)], step=0), 1, b"step"),
        (lambda: commit([fake(8, p=2)]), 2, b"aligned"),
        (lambda: commit([fake(100, goff=M64 - 50)]), 3, b"overflow"),
        (lambda: lib.apc_set_reserved_sms(-3), 1, b"reserved"),
    ]
    failures = []

    def run(k):
        call, status, word = cases[k % len(cases)]
        for _ in range(200):
            st = call()
            msg = lib.apc_last_error()
            if st != status or word not in msg.lower():
                failures.append((k, st, msg))
                return

    threads = [threading.Thread(target=run, args=(k,)) for k in range(8)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    assert not failures, failures[:3]
