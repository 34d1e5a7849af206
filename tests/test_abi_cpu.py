"""CPU checks of the C ABI: the library builds, loads, and exports every entry
point include/malib.h declares; without a GPU, context creation fails with a
status code instead of crashing. No compute call is made here."""
import ctypes as C
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_symbols():
    text = open(os.path.join(ROOT, "include", "malib.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(malib_[a-z_0-9]+)\s*\(", text)))


@pytest.fixture(scope="module")
def libpath():
    from paper_2106_07551_gb300 import build
    return build.build()


def test_header_and_binding_agree():
    from paper_2106_07551_gb300 import _abi
    assert declared_symbols() == sorted(_abi.EXPORTS)


def test_library_exports_every_declared_symbol(libpath):
    out = subprocess.run(["nm", "-D", "--defined-only", libpath], capture_output=True, text=True,
                         check=True).stdout
    exported = set(re.findall(r"\bT (malib_\w+)", out))
    missing = [s for s in declared_symbols() if s not in exported]
    assert not missing, missing


def test_binding_loads_and_create_fails_cleanly_without_gpu(libpath):
    import torch
    from paper_2106_07551_gb300 import _abi, MalibError, malib_create
    lib = _abi.load(libpath)
    for name in _abi.EXPORTS:
        assert hasattr(lib, name)
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    h = C.c_void_p()
    code = lib.malib_create(C.byref(h), 0, None)
    assert code in (_abi.MALIB_ECUDA, _abi.MALIB_EINVAL)
    assert not h.value
    assert lib.malib_last_error(None)
    with pytest.raises(MalibError):
        malib_create(0)
    # null context: every call reports EINVAL, none touches a GPU
    assert lib.malib_sync(None) == _abi.MALIB_EINVAL
    assert lib.malib_eval_payoff(None, None, 0, 1, 0, None) == _abi.MALIB_EINVAL
    assert lib.malib_launch_count(None) == 0


def test_missing_library_fails_loudly(tmp_path):
    from paper_2106_07551_gb300 import _abi
    if _abi._lib is not None:
        saved, _abi._lib = _abi._lib, None
    else:
        saved = None
    try:
        with pytest.raises(ImportError):
            _abi.load(str(tmp_path / "nope.so"))
    finally:
        _abi._lib = saved


def test_env_spec_layout_and_local_ratio_flag():
    """The spec's last field is the spread reward's local_ratio (a float in the
    slot of the same size); make_spec sets the flag only when it is given."""
    import ctypes as C
    from paper_2106_07551_gb300 import _abi, make_spec
    assert C.sizeof(_abi.EnvSpec) == 40
    assert _abi.EnvSpec.local_ratio.offset == 36
    s = make_spec(3, 3, 18, 5, 3, 25, 4096)
    assert s.flags & _abi.MALIB_SPREAD_LOCAL_RATIO == 0
    s = make_spec(3, 3, 18, 5, 3, 25, 4096, local_ratio=0.25)
    assert s.flags & _abi.MALIB_SPREAD_LOCAL_RATIO and abs(s.local_ratio - 0.25) < 1e-7
