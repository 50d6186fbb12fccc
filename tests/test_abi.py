"""The C-ABI library builds, loads without a GPU and exports every symbol that
include/ffh.h declares; the Python options struct matches the header's layout.
No compute call is made here."""
import ctypes
import re

import pytest

import paper_2609_14706_gb300 as ffh
from paper_2609_14706_gb300 import build as ffh_build


@pytest.fixture(scope="module")
def lib():
    ffh_build.build()
    return ffh.load_library()


def test_exports_every_declared_symbol(lib):
    names = ffh.header_symbols()
    assert len(names) >= 12
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing


def test_version(lib):
    assert lib.ffh_version() >= 100


def test_options_struct_layout_matches_header():
    text = open(ffh.HEADER_PATH).read()
    body = re.search(r"typedef struct \{(.*?)\} ffh_options;", text, re.S).group(1)
    body = re.sub(r"/\*.*?\*/", "", body, flags=re.S)
    fields = re.findall(r"\b(\w+)\s*(?:\[\d+\])?;", body)
    assert fields == [f for f, _ in ffh.ffh_options._fields_]
    assert ctypes.sizeof(ffh.ffh_options) == 56


def test_status_codes_match_header():
    text = open(ffh.HEADER_PATH).read()
    for code, name in ffh.STATUS.items():
        assert re.search(rf"\b{name}\s*=\s*{code}\b", text), name


def test_null_handle_calls_are_rejected(lib):
    assert lib.ffh_destroy(None) == 0
    assert lib.ffh_fit(None, None, None, 1, 1, 1, 1, 0.0, None, None) == 1
    assert lib.ffh_last_error(None) == b"null handle"
