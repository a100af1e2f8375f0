"""The C ABI: libsoap.so loads without a GPU, exports every function include/soap.h declares,
and rejects invalid arguments on the host before touching the device."""
import ctypes
import os
import re

from paper_2607_20548_gb300 import build
from paper_2607_20548_gb300 import soap as S

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared(header="soap.h", prefix="soap_"):
    text = open(os.path.join(ROOT, "include", header)).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(" + prefix + r"[a-z0-9_]+)\s*\(", text)))


def test_library_exports_every_declared_symbol():
    build.build()
    lib = S.load_library()
    names = _declared()
    assert "soap_create" in names and "soap_step" in names and "soap_state_get" in names
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing
    assert set(names) == set(S.EXPORTS)
    muon = _declared("muon.h", "muon_")
    assert "muon_create" in muon and "muon_step" in muon
    assert not [n for n in muon if not hasattr(lib, n)]
    assert set(muon) == set(S.MUON_EXPORTS)


def test_host_side_validation_needs_no_gpu():
    lib = S.load_library()
    h = ctypes.c_void_p()
    hp = S.soap_hparams()
    lib.soap_default_hparams(ctypes.byref(hp))
    assert abs(hp.lr - 3e-3) < 1e-9 and hp.eig_every == 1 and abs(hp.qr_tol - 2e-5) < 1e-9
    shapes = (S.soap_shape * 1)(S.soap_shape(0, 5, 1, 1))
    assert lib.soap_create(shapes, 1, ctypes.byref(hp), 0, ctypes.byref(h)) == 1
    assert not h.value
    big = (S.soap_shape * 1)(S.soap_shape(10000, 5, 1, 1))  # preconditioned side > 8192
    assert lib.soap_create(big, 1, ctypes.byref(hp), 0, ctypes.byref(h)) == 1
    bad_hp = S.soap_hparams()
    lib.soap_default_hparams(ctypes.byref(bad_hp))
    bad_hp.eig_every = 0
    ok_shape = (S.soap_shape * 1)(S.soap_shape(4, 5, 1, 1))
    assert lib.soap_create(ok_shape, 1, ctypes.byref(bad_hp), 0, ctypes.byref(h)) == 1
    # the KL-Shampoo factor form is off by default and needs eps > 0 (its first step weighs by 1/eps)
    assert hp.kl == 0
    kl_hp = S.soap_hparams()
    lib.soap_default_hparams(ctypes.byref(kl_hp))
    kl_hp.kl, kl_hp.eps = 1, 0.0
    assert lib.soap_create(ok_shape, 1, ctypes.byref(kl_hp), 0, ctypes.byref(h)) == 1
    kl_hp.kl, kl_hp.eps = 2, 1e-8
    assert lib.soap_create(ok_shape, 1, ctypes.byref(kl_hp), 0, ctypes.byref(h)) == 1
    # the stale variant needs the guard off and the standard factor form
    assert hp.stale == 0
    st_hp = S.soap_hparams()
    lib.soap_default_hparams(ctypes.byref(st_hp))
    st_hp.stale = 1
    assert lib.soap_create(ok_shape, 1, ctypes.byref(st_hp), 0, ctypes.byref(h)) == 1
    st_hp.guard, st_hp.kl = 0, 1
    assert lib.soap_create(ok_shape, 1, ctypes.byref(st_hp), 0, ctypes.byref(h)) == 1
    assert lib.soap_gemm(0, 0, -1, 1, 1, 1.0, None, 1, 0, None, 1, 0, 0.0, None, 1, 0, 1, None) == 1
    assert lib.soap_gemm(0, 0, 0, 1, 1, 1.0, None, 1, 0, None, 1, 0, 0.0, None, 1, 0, 1, None) == 0
    assert lib.soap_qr(0, 1, None, None, None, 0.0, None, 0, None, None) == 1
    assert lib.soap_qr_workspace_bytes(64, 2) > 2 * 64 * 64 * 4
    assert lib.soap_state_bytes(None, 0, 0) == 0
    assert lib.soap_get_step(None) == -1
    assert lib.soap_last_error(None) == b"null handle"
    lib.soap_destroy(None)
    # profiling: a null handle, and (checked before any device work) unknown flags, are refused
    assert lib.soap_profile_begin_ex(None, 16, S.PROFILE_SERIAL) == 1
    assert lib.soap_profile_records(None, None, 0, None) == 1
    assert ctypes.sizeof(S.soap_launch_record) == 40  # int32 family (padded), start, end, flops, bytes
    # Muon: sides must be multiples of 8, ns_steps in 1..64
    mh = S.muon_hparams()
    lib.muon_default_hparams(ctypes.byref(mh))
    assert mh.ns_steps == 16 and abs(mh.beta1 - 0.9) < 1e-7 and abs(mh.eps - 1e-7) < 1e-12
    bad = (S.soap_shape * 1)(S.soap_shape(12, 16, 0, 0))
    assert lib.muon_create(bad, 1, ctypes.byref(mh), 0, ctypes.byref(h)) == 1
    mh.ns_steps = 0
    good = (S.soap_shape * 1)(S.soap_shape(16, 16, 0, 0))
    assert lib.muon_create(good, 1, ctypes.byref(mh), 0, ctypes.byref(h)) == 1
    assert lib.muon_last_error(None) == b"null handle"
    lib.muon_destroy(None)


def test_missing_library_fails_loudly():
    """Without libsoap.so the binding raises; there is no other path that computes the step."""
    import pytest
    saved = S._lib
    S._lib = None
    try:
        with pytest.raises(ImportError, match="libsoap.so not built"):
            S.load_library(os.path.join(ROOT, "no_such_dir", "libsoap.so"))
    finally:
        S._lib = saved


def test_product_code_shares_nothing_with_the_oracle():
    """The package (binding, workloads, CUDA sources) neither imports nor includes anything from
    oracle/; only tests, the smoke entry and the bench's CPU baseline use the oracle."""
    pkg = os.path.join(ROOT, "paper_2607_20548_gb300")
    pat = re.compile(r"^\s*(from\s+oracle\b|import\s+oracle\b|#\s*include\s*[<\"][^>\"]*oracle)", re.M)
    offenders = []
    for dirpath, _, files in os.walk(pkg):
        if "_build" in dirpath or "_lib" in dirpath or "__pycache__" in dirpath:
            continue
        for f in files:
            if f.endswith((".py", ".cu", ".h", ".cuh", ".cpp", ".c")):
                text = open(os.path.join(dirpath, f)).read()
                if pat.search(text):
                    offenders.append(f)
    assert not offenders, offenders
    for f in os.listdir(os.path.join(ROOT, "oracle")):
        if f.endswith((".py", ".c", ".h")):
            text = open(os.path.join(ROOT, "oracle", f)).read()
            assert "paper_2607_20548_gb300" not in text and "csrc" not in text, f


class _FakeCudaTensor:
    """Just enough of a CUDA tensor for the binding's argument checks (never reaches the library)."""

    def __init__(self, shape, index):
        import torch
        self.shape, self.dtype, self.is_cuda = shape, torch.float32, True
        self.device = torch.device("cuda", index)

    def is_contiguous(self):
        return True

    def data_ptr(self):
        return 1 << 20


def test_binding_rejects_tensors_on_another_device():
    """A handle steps tensors on its own device only; the check happens before any library call."""
    import ctypes as ct

    import pytest
    for cls in (S.SoapOptimizer, S.MuonOptimizer):
        opt = cls.__new__(cls)
        opt.shapes = [S.Shape(4, 8)] if cls is S.SoapOptimizer else [(4, 8)]
        opt.device, opt._h = 0, None
        opt._pp, opt._gp = (ct.c_void_p * 1)(), (ct.c_void_p * 1)()
        with pytest.raises(ValueError, match="cuda:0"):
            opt.step([_FakeCudaTensor((4, 8), 1)], [_FakeCudaTensor((4, 8), 1)])
        with pytest.raises(ValueError, match="cuda:0"):
            opt.step([_FakeCudaTensor((4, 8), 0)], [_FakeCudaTensor((4, 8), 1)])
        # tensors on the handle's device pass the checks (and reach the handle, destroyed here)
        with pytest.raises(S.SoapError, match="handle destroyed"):
            opt.step([_FakeCudaTensor((4, 8), 0)], [_FakeCudaTensor((4, 8), 0)])


def test_standalone_entry_points_reject_host_tensors():
    """The stand-alone sub-steps hand only CUDA tensors of the right type to the kernels: host
    tensors are refused on the host, before any launch."""
    import pytest
    import torch
    x = torch.zeros(4, 4)
    for call in (lambda: S.soap_gemm(x, x), lambda: S.soap_split_tf32(x), lambda: S.soap_gemm_tf32x4(x, x),
                 lambda: S.soap_qr(x), lambda: S.soap_qr_static(x)):
        with pytest.raises(TypeError):
            call()


def test_plain_c_consumer_builds_and_runs():
    """include/*.h are plain C: a C99 program compiles against them with gcc alone, links
    libsoap.so and runs its host-side entry points."""
    import shutil
    import subprocess
    import tempfile

    import pytest
    if shutil.which("gcc") is None:
        pytest.skip("no gcc")
    lib = build.build()
    with tempfile.TemporaryDirectory() as d:
        exe = os.path.join(d, "c_abi_host")
        r = subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"),
                            os.path.join(ROOT, "tests", "c_abi_host.c"), lib, "-Wl,-rpath," + os.path.dirname(lib),
                            "-o", exe], capture_output=True, text=True)
        assert r.returncode == 0, r.stderr
        r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
        assert r.returncode == 0 and "c abi ok" in r.stdout, (r.returncode, r.stdout, r.stderr)


def test_stream_of_another_device_is_refused():
    """A caller's stream must belong to the device the work runs on: one of another device is
    refused on the host with a clear error instead of reaching the library."""
    import pytest
    import torch

    class _FakeStream:
        def __init__(self, index):
            self.device = torch.device("cuda", index)
            self.cuda_stream = 0

    assert S._stream(_FakeStream(1), 1).value in (0, None)
    with pytest.raises(ValueError):
        S._stream(_FakeStream(1), 0)
    with pytest.raises(ValueError):
        S._stream(_FakeStream(0), torch.device("cuda", 2))
