"""Host-side checks of the C-ABI library (no GPU needed): it loads, exports
every entry point include/pvmvmd.h declares, resolves the paper's parameters,
rejects bad arguments before touching a device, and its host sampler of the
public codes agrees bit for bit with the oracle's."""
import ctypes
import json
import os
import re

import numpy as np
import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "pvmvmd.h")


@pytest.fixture(scope="module")
def pv():
    import __graft_entry__
    __graft_entry__._load_build_module().build()
    import paper_2609_10264_gb300 as pv
    return pv


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(pvmvmd_[a-z_]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(pv):
    names = _declared()
    assert "pvmvmd_server_mvm" in names and "pvmvmd_encode" in names
    lib = ctypes.CDLL(pv.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n
        assert n in pv.SIGNATURES, n


def test_strerror(pv):
    codes = [pv.PVMVMD_OK, pv.PVMVMD_E_ARG, pv.PVMVMD_E_SHAPE, pv.PVMVMD_E_PARAM, pv.PVMVMD_E_CUDA,
             pv.PVMVMD_E_NOMEM, pv.PVMVMD_E_DEVICE_TIMEOUT, pv.PVMVMD_E_NODEVICE]
    msgs = [pv.pvmvmd_strerror(c) for c in codes]
    assert len(set(msgs)) == len(codes)
    assert pv.pvmvmd_strerror(-99) == "unknown status"


def test_params_default_to_the_paper(pv):
    g = json.load(open(os.path.join(ROOT, "tests", "golden", "paper_params.json")))
    for n, t in zip(g["t_x_by_n"]["n"], g["t_x_by_n"]["t_x"]):
        p = pv.pvmvmd_params_resolve(n, n)
        assert (p.t_x, p.t_y, p.ell, p.rate, p.lambda_, p.kappa) == (t, 31, 2, 8, 128, 40)
        assert p.delta == 0.5
    for K in (1, 7, 256, 4096, 14336, 28672, 131071):
        assert pv.pvmvmd_params_resolve(64, K).t_x == oracle.t_x(K) if K * 8 >= 163 else True


def test_params_overrides_and_errors(pv):
    p = pv.pvmvmd_params()
    p.t_x, p.t_y, p.ell, p.rate = 5, 3, 1, 4
    r = pv.pvmvmd_params_resolve(10, 10, p)
    assert (r.t_x, r.t_y, r.ell, r.rate) == (5, 3, 1, 4)
    bad = pv.pvmvmd_params()
    bad.t_x = 81  # N_x = 8 * 10 = 80
    with pytest.raises(pv.PvmvmdError) as e:
        pv.pvmvmd_params_resolve(10, 10, bad)
    assert e.value.status == pv.PVMVMD_E_PARAM
    bad = pv.pvmvmd_params()
    bad.t_y = 81
    with pytest.raises(pv.PvmvmdError):
        pv.pvmvmd_params_resolve(10, 10, bad)
    bad = pv.pvmvmd_params()
    bad.delta = 1.5
    with pytest.raises(pv.PvmvmdError):
        pv.pvmvmd_params_resolve(10, 10, bad)
    # Eq. (1) asks for t_x = 174 at K = 1 (N_x = 8): more than N_x
    with pytest.raises(pv.PvmvmdError):
        pv.pvmvmd_params_resolve(64, 1)


def test_bad_arguments_rejected_before_device_use(pv):
    lib = pv._lib
    vp = ctypes.c_void_p
    assert lib.pvmvmd_server_mvm(None, 4, 4, None, 1, None, None) == pv.PVMVMD_E_ARG
    one = vp(16)  # never dereferenced: the shape check fails first
    assert lib.pvmvmd_server_mvm(one, 0, 4, one, 1, one, None) == pv.PVMVMD_E_SHAPE
    assert lib.pvmvmd_server_mvm(one, 4, pv.PVMVMD_MAX_K + 1, one, 1, one, None) == pv.PVMVMD_E_SHAPE
    assert lib.pvmvmd_server_mvm(one, 4, 4, one, 0, one, None) == pv.PVMVMD_E_SHAPE
    out = vp()
    assert lib.pvmvmd_preprocess(None, 4, 4, None, None, None, ctypes.byref(out)) == pv.PVMVMD_E_ARG
    assert out.value is None
    assert lib.pvmvmd_encode(None, one, 1, None, one, one, None) == pv.PVMVMD_E_ARG
    assert lib.pvmvmd_decode_verify(None, one, one, one, 1, None, one, one, None) == pv.PVMVMD_E_ARG
    assert lib.pvmvmd_ctx_info(None, None) == pv.PVMVMD_E_ARG
    nbytes = ctypes.c_size_t()
    assert lib.pvmvmd_code_encode_scratch(None, 0, 4, ctypes.byref(nbytes)) == pv.PVMVMD_E_ARG
    assert lib.pvmvmd_code_encode_scratch(one, 2, 4, ctypes.byref(nbytes)) == pv.PVMVMD_E_ARG
    assert lib.pvmvmd_code_encode_lanes(one, 0, one, 4, None, one, None) == pv.PVMVMD_E_ARG
    assert lib.pvmvmd_code_encode_lanes(one, -1, one, 4, one, one, None) == pv.PVMVMD_E_ARG
    lib.pvmvmd_destroy(None)


@pytest.mark.parametrize("which,N,seed", [(0, 8, 0), (1, 8, 5), (0, 2048, 1), (1, 32776, 2),
                                          (0, 114688, 3)])
def test_host_code_sampler_matches_oracle(pv, which, N, seed):
    lib_tables = pv.pvmvmd_code_sample_host(seed, which, N)
    orc = oracle.Code.sample(oracle.key_from_seed(seed), which, N // 8, 8)
    for a, b in zip(lib_tables, (orc.pi1, orc.pi2, orc.v1, orc.v2)):
        assert np.array_equal(a, b)


def test_key_conventions_agree(pv):
    s = (5 << 200) | (7 << 33) | 11
    k = pv.make_key(s)
    assert list(k.k) == oracle.key_from_seed(s).tolist()
    assert list(pv.make_key(bytes(range(32))).k) == list(np.frombuffer(bytes(range(32)), "<u4"))


def test_input_generators_map_no_cuda_library():
    """The seeded input generators (which the oracle arm of the bench and the
    oracle tests use) load without opening libpvmvmd.so: the package opens it
    only on its first call."""
    import subprocess
    import sys
    code = ("import sys; sys.path.insert(0, %r)\n"
            "from paper_2609_10264_gb300 import workloads\n"
            "workloads.weights_gaussian(4, 8, 0)\n"
            "maps = open('/proc/self/maps').read()\n"
            "assert 'libpvmvmd' not in maps, 'library mapped at import'\n"
            "import paper_2609_10264_gb300 as pv\n"
            "assert pv.pvmvmd_strerror(0) == 'success'\n"
            "assert 'libpvmvmd' in open('/proc/self/maps').read()\n") % ROOT
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr


def test_debug_wait_hook_arguments(pv):
    """The failure-path test hook is host-only state: it rejects unknown sites
    and zero limits, and switches off cleanly."""
    lib = pv._lib
    assert lib.pvmvmd_debug_expire_wait(7, 0, 1) == pv.PVMVMD_E_ARG
    assert lib.pvmvmd_debug_expire_wait(pv.PVMVMD_DEBUG_WAIT_SCAN, 0, 0) == pv.PVMVMD_E_ARG
    assert lib.pvmvmd_debug_expire_wait(pv.PVMVMD_DEBUG_WAIT_PRODUCT, 3, 1000) == pv.PVMVMD_OK
    assert lib.pvmvmd_debug_expire_wait(pv.PVMVMD_DEBUG_WAIT_OFF, 0, 0) == pv.PVMVMD_OK
