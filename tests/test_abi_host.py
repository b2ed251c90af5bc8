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


def test_binding_fails_loudly_without_the_library(tmp_path):
    # a copy of the binding beside no built library: importing it raises
    # instead of falling back to anything else
    import importlib.util
    import shutil
    src = os.path.join(ROOT, "paper_2607_13093_gb300", "sph.py")
    dst = tmp_path / "sph_copy.py"
    shutil.copy(src, dst)
    spec = importlib.util.spec_from_file_location("sph_copy", dst)
    mod = importlib.util.module_from_spec(spec)
    with pytest.raises(RuntimeError, match="not built"):
        spec.loader.exec_module(mod)


def test_product_package_never_imports_the_oracle():
    pkg = os.path.join(ROOT, "paper_2607_13093_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h", ".cpp", ".c")):
                text = open(os.path.join(dirpath, f), errors="replace").read()
                assert not re.search(r"^\s*(import|from)\s+oracle\b", text, flags=re.M), f
                assert "sph_oracle" not in text, f


def test_oracle_imports_nothing_of_the_product():
    # the oracle depends on numpy alone (and on its own modules)
    import ast
    odir = os.path.join(ROOT, "oracle")
    for f in os.listdir(odir):
        if f.endswith(".py"):
            tree = ast.parse(open(os.path.join(odir, f)).read())
            for node in ast.walk(tree):
                if isinstance(node, ast.Import):
                    mods = [a.name for a in node.names]
                elif isinstance(node, ast.ImportFrom):
                    if node.level > 0:
                        continue
                    mods = [node.module]
                else:
                    continue
                for m in mods:
                    assert m.split(".")[0] in ("numpy", "__future__"), (f, m)


def test_check_keep_ids_against_the_conventions(sph):
    # strictly increasing ids in [0, V): the first offending position is
    # reported (host lists only; nothing here reaches a kernel)
    ok = np.array([0, 3, 4, 9], np.int32)
    assert sph.sph_check_keep_ids(ok, 10) == (True, -1)
    assert sph.sph_check_keep_ids(ok, 9) == (False, 3)            # id == V
    assert sph.sph_check_keep_ids([0, 3, 3, 9], 10) == (False, 2)  # repeated
    assert sph.sph_check_keep_ids([0, 5, 4, 9], 10) == (False, 2)  # unsorted
    assert sph.sph_check_keep_ids([-1, 5], 10) == (False, 0)       # negative
    assert sph.sph_check_keep_ids([7], 8) == (True, -1)
    assert not sph.sph_check_keep_ids(np.zeros(0, np.int32), 8)[0]
    rng = np.random.default_rng(3)
    for _ in range(20):
        V = int(rng.integers(2, 500))
        ids = np.sort(rng.choice(V, size=int(rng.integers(1, V)), replace=False))
        assert sph.sph_check_keep_ids(ids, V) == (True, -1)
        bad = ids.copy()
        j = int(rng.integers(0, ids.size))
        bad[j] = V + int(rng.integers(0, 3))
        good, at = sph.sph_check_keep_ids(bad, V)
        assert not good and at <= j


def test_binding_refuses_buffers_the_kernels_would_leave(sph):
    # the kernels index codes, scales, tokens, fused logits, id lists and
    # the verification's inputs densely: the binding refuses a buffer that
    # is on another device, strided, or smaller than the call needs, before
    # anything reaches the library; operands with a row stride are checked
    # for their device only
    import torch
    cpu = torch.device("cpu")
    ok = torch.empty(4, 300)
    sph._dense(cpu, (ok, "z", 4 * 300), (torch.empty(5, 300), "bigger", 4 * 300),
               (None, "absent", 10), (torch.empty(4, 600)[:, :300], "W", None),
               (torch.empty(2, 0), "empty", 0))
    bad = [(torch.empty(4, 300, device="meta"), 4 * 300, "not on"),
           (torch.empty(4, 8, device="meta")[:, :4], None, "not on"),
           (torch.empty(300, 4).t(), 4 * 300, "contiguous"),
           (torch.empty(8)[::2], 4, "contiguous"),
           (torch.empty(3, 300), 4 * 300, "elements")]
    for t, count, what in bad:
        with pytest.raises(ValueError, match=what):
            sph._dense(cpu, (t, "x", count))


def test_binding_constants_match_the_header(sph):
    # every option, activation mode and weight type the binding mirrors has
    # the header's value, every option of the header is mirrored, and every
    # option name bench.py accepts (--opt NAME=VALUE) resolves to one of them
    import bench
    text = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    header = {m.group(1): int(m.group(2))
              for m in re.finditer(r"\b(SPH_[A-Z0-9_]+)\s*=\s*(\d+)", text)}
    mirrored = {k: v for k, v in vars(sph).items()
                if k.startswith(("SPH_OPT_", "SPH_ACT_", "SPH_DTYPE_")) and isinstance(v, int)}
    assert mirrored
    for name, value in mirrored.items():
        assert header.get(name) == value, (name, value, header.get(name))
    options = {k for k in header if k.startswith("SPH_OPT_")}
    assert options == {k for k in mirrored if k.startswith("SPH_OPT_")}
    assert set(bench.OPTION_NAMES.values()) <= options


def test_binding_structs_and_signatures_follow_the_header(sph):
    # the ctypes mirrors of sph_plan and sph_profile have the header's
    # fields in its order and types, and every bound function takes as many
    # arguments as the header declares
    import ctypes
    text = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)

    def struct_fields(name):
        body = re.search(r"typedef struct %s \{(.*?)\}" % name, text, flags=re.S).group(1)
        return re.findall(r"(\w+)\s+(\w+)(?:\[(\w+)\])?\s*;", body)

    assert [(t, f) for t, f, _ in struct_fields("sph_plan")] == \
        [("int32_t", f) for f in sph.PLAN_FIELDS]
    assert [f for f, _ in sph.sph_plan._fields_] == list(sph.PLAN_FIELDS)
    n_classes = int(re.search(r"\bSPH_PROF_CLASSES\s*=\s*(\d+)", text).group(1))
    assert sph.PROF_CLASSES == n_classes
    assert struct_fields("sph_profile") == [("double", "ms", "SPH_PROF_CLASSES"),
                                            ("int64_t", "calls", "SPH_PROF_CLASSES"),
                                            ("int64_t", "launches", "")]
    assert [(f, t) for f, t in sph.sph_profile._fields_] == [
        ("ms", ctypes.c_double * n_classes), ("calls", ctypes.c_int64 * n_classes),
        ("launches", ctypes.c_int64)]
    for fn, (_, argtypes) in sph._SIGNATURES.items():
        m = re.search(r"\b%s\s*\(([^)]*)\)\s*;" % fn, text)
        assert m, fn
        params = [p for p in m.group(1).split(",") if p.strip() and p.strip() != "void"]
        assert len(params) == len(argtypes), (fn, len(params), len(argtypes))
