"""The C ABI library loads and exports every symbol include/gleam.h declares,
and rejects bad arguments before touching the GPU.  No compute call is made."""
import ctypes
import os
import re
import subprocess

import pytest

from paper_2607_23115_gb300 import binding as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "gleam.h")


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(gleam_[a-z0-9_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    from paper_2607_23115_gb300 import build
    build.build()
    return B.lib()


def test_header_declarations_match_binding():
    assert _declared() == sorted(B.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    for name in _declared():
        assert hasattr(lib, name), name
    out = subprocess.run(["nm", "-D", "--defined-only", B.LIB_PATH], capture_output=True,
                         text=True).stdout
    for name in _declared():
        assert re.search(r"\sT\s%s$" % name, out, flags=re.M), name


def test_status_strings(lib):
    assert B.gleam_status_string(B.GLEAM_ERR_CAPACITY) == "cache capacity exceeded"
    assert B.gleam_status_string(12345) == "unknown status"


@pytest.mark.parametrize("cap,chunk,flags", [
    (1 << 20, 0, 0), (1 << 20, 33, 0), (1 << 20, 16, 0), (1 << 20, 32 << 20, 0),
    (100, 1024, 0), (1 << 20, 1024, 0x80), ((1 << 32) * 64, 32, 0)])
def test_create_rejects_bad_arguments_without_a_gpu(lib, cap, chunk, flags):
    rc, h = B.gleam_cache_create_ex(cap, chunk, flags)
    assert rc == B.GLEAM_ERR_INVALID_ARG and h is None


def test_null_handles_are_rejected(lib):
    assert B.gleam_dedup_copy(None, None, 10, None, None, None) == B.GLEAM_ERR_INVALID_ARG
    assert B.gleam_dedup_copy_async(None, None, 10, None, None, None) == B.GLEAM_ERR_INVALID_ARG
    assert B.gleam_cache_stats(None)[0] == B.GLEAM_ERR_INVALID_ARG
    assert B.gleam_fingerprint(None, 10, 64, None) == B.GLEAM_ERR_INVALID_ARG
    B.gleam_cache_destroy(None)


def test_gleam_struct_sizes():
    """The binding's structs have the header's fields, in the header's order."""
    with open(HEADER) as f:
        h = f.read()
    body = re.search(r"typedef struct gleam_stats \{(.*?)\} gleam_stats_t;", h, re.S).group(1)
    fields = re.findall(r"uint64_t (\w+);", body)
    assert [f for f, _ in B.gleam_stats_t._fields_] == fields
    assert ctypes.sizeof(B.gleam_stats_t) == 8 * len(fields)
    assert B.RESULT_WORDS * 8 == 48
