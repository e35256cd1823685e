"""CPU-side checks of the C ABI: the library builds, loads without a GPU, exports every
entry point include/c2kv.h declares, and its host-side argument checks answer before
any CUDA call.  No compute runs here."""
import os
import re
import subprocess

import pytest


@pytest.fixture(scope="module")
def c2kv(repo_root):
    import __graft_entry__ as g
    g.build()
    from paper_2607_17715_gb300 import c2kv as mod
    return mod


def _declared(repo_root):
    names = set()
    for fn in os.listdir(os.path.join(repo_root, "include")):
        if fn.endswith(".h"):
            src = open(os.path.join(repo_root, "include", fn)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(c2kv_\w+)\s*\(", src))
    return names


def test_header_declares_the_boundary(repo_root):
    names = _declared(repo_root)
    for must in ("c2kv_compress_chunk", "c2kv_compose", "c2kv_attend", "c2kv_create",
                 "c2kv_destroy", "c2kv_sync", "c2kv_last_error"):
        assert must in names


def test_library_exports_every_declared_symbol(c2kv, repo_root):
    out = subprocess.run(["nm", "-D", "--defined-only", c2kv.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = {ln.split()[-1] for ln in out.splitlines() if " T " in ln}
    missing = _declared(repo_root) - exported
    assert not missing, f"declared but not exported: {sorted(missing)}"
    for name in _declared(repo_root):
        assert hasattr(c2kv._lib, name)


def test_binding_names_match_header(c2kv, repo_root):
    for name in _declared(repo_root):
        assert hasattr(c2kv, name), f"binding lacks {name}"


def test_abi_version(c2kv):
    assert c2kv.c2kv_abi_version() == 5


@pytest.mark.parametrize("args,status", [
    ((0, 4, 2, 64, 1e4, 1, 16), -1),        # layers
    ((1, 4, 3, 64, 1e4, 1, 16), -1),        # Hq % Hkv
    ((1, 4, 2, 96, 1e4, 1, 16), -1),        # head_dim
    ((1, 4, 2, 64, 0.5, 1, 16), -1),        # theta
    ((1, 4, 2, 64, 1e4, 5, 16), -2),        # dtype
    ((1, 4, 2, 64, 1e4, 1, 0), -1),         # pool
])
def test_create_validates_before_cuda(c2kv, args, status):
    with pytest.raises(c2kv.C2KVError) as ei:
        c2kv.c2kv_create(*args)
    assert ei.value.status == status
    assert c2kv.c2kv_last_error(None)


def test_null_handles(c2kv):
    assert c2kv._lib.c2kv_sync(None) == c2kv.ERR_ARG
    assert c2kv._lib.c2kv_destroy(None) == c2kv.OK
    assert c2kv._lib.c2kv_compose(None, 1, None, None, None, 0, None) == c2kv.ERR_ARG
    assert c2kv._lib.c2kv_attend(None, None, 0, None, None, None, 1, None, None) == c2kv.ERR_ARG
