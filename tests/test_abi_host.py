"""The C-ABI library builds, loads and exports every symbol of include/sph.h;
host-only helpers agree with plain definitions (no GPU needed)."""
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "sph.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(sph_[a-z0-9_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def sph():
    from paper_2607_13093_gb300 import build_lib
    build_lib.build()
    from paper_2607_13093_gb300 import sph as mod
    return mod


def test_header_declares_the_hot_path():
    names = declared_functions()
    for must in ("sph_partial_logits", "sph_fuse_sample", "sph_verify_draft",
                 "sph_create", "sph_destroy", "sph_set_stream", "sph_sync",
                 "sph_buffer_alloc", "sph_buffer_free", "sph_buffer_ptr"):
        assert must in names


def test_every_declared_symbol_is_exported(sph):
    for name in declared_functions():
        assert hasattr(sph.lib, name), name
    out = os.popen(f"nm -D --defined-only {sph.LIB_PATH}").read()
    exported = set(re.findall(r"\bT (sph_[a-z0-9_]+)", out))
    assert set(declared_functions()) <= exported


def test_binding_covers_every_symbol(sph):
    assert set(declared_functions()) == set(sph._SIGNATURES)


def test_payload_bytes_matches_eq21(sph):
    import oracle
    for rows, n in [(1, 150000), (32, 12000), (320, 51302), (0, 5)]:
        assert sph.sph_payload_bytes(rows, n) == oracle.payload_bytes(rows, n)
    assert sph.lib.sph_payload_bytes(-1, 5) == 0


def test_keep_ids_from_mask(sph):
    rng = np.random.default_rng(0)
    for V in (1, 7, 8, 9, 1000, 8193):
        keep = rng.random(V) < 0.3
        keep[rng.integers(0, V)] = True
        bits = np.packbits(keep, bitorder="little")
        ids = sph.sph_keep_ids_from_mask(bits, V)
        assert ids.dtype == np.int32
        assert np.array_equal(ids, np.nonzero(keep)[0])
    with pytest.raises(sph.SphError):
        sph.sph_keep_ids_from_mask(np.zeros(2, np.uint8), 16)


def test_status_strings(sph):
    for code, name in sph.STATUS_NAMES.items():
        assert sph.lib.sph_status_string(code).decode() == name


def test_create_without_device_fails_cleanly(sph):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    with pytest.raises(sph.SphError):
        sph.sph_create(0, None)
