"""The library build is keyed on content: a changed flag or source recompiles, an unchanged tree reuses
its objects, and an object whose bytes no longer match its recorded hash (one carried over from another
build, whatever its time stamp) is compiled again.  CPU only (nvcc cross-compiles for sm_103a)."""
import os
import shutil

import pytest

from paper_2609_22158_gb300 import build as BLD

pytestmark = pytest.mark.skipif(shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"),
                                reason="nvcc not available")


def test_rebuild_follows_content_not_mtime(tmp_path):
    bdir, lib = str(tmp_path / "b"), str(tmp_path / "libprobe.so")
    log = []
    src = ["decode.cu"]
    BLD.build_library(build_dir=bdir, lib_path=lib, sources=src, log=log)
    assert log[-1]["compiled"] == ["decode.cu"] and log[-1]["linked"]
    key0 = log[-1]["library_key"]
    assert len(key0) == 16

    BLD.build_library(build_dir=bdir, lib_path=lib, sources=src, log=log)
    assert log[-1]["compiled"] == [] and not log[-1]["linked"] and log[-1]["library_key"] == key0

    # a changed flag changes the key and recompiles
    BLD.build_library(build_dir=bdir, lib_path=lib, sources=src, log=log, extra_flags=["-DSTEPKV_BUILD_PROBE=1"])
    assert log[-1]["compiled"] == ["decode.cu"] and log[-1]["linked"] and log[-1]["library_key"] != key0

    # an object replaced behind the build's back (newer time stamp, same key file) is not reused
    obj = os.path.join(bdir, "decode.o")
    with open(obj, "ab") as f:
        f.write(b"\0")
    st = os.stat(obj)
    os.utime(obj, (st.st_atime + 3600, st.st_mtime + 3600))
    BLD.build_library(build_dir=bdir, lib_path=lib, sources=src, log=log, extra_flags=["-DSTEPKV_BUILD_PROBE=1"])
    assert log[-1]["compiled"] == ["decode.cu"]

    # a library replaced behind the build's back is relinked
    with open(lib, "ab") as f:
        f.write(b"\0")
    BLD.build_library(build_dir=bdir, lib_path=lib, sources=src, log=log, extra_flags=["-DSTEPKV_BUILD_PROBE=1"])
    assert log[-1]["compiled"] == [] and log[-1]["linked"]
