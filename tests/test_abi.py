"""The C-ABI library loads, exports what include/*.h declares, and rejects
bad arguments on the host before any launch (no GPU needed, no compute)."""
import ctypes
import glob
import os
import re

import pytest

from paper_2607_20214_gb300 import build, elsaa
from paper_2607_20214_gb300.workloads import WORKLOADS

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return elsaa.load_library()


def declared_functions():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        src = re.sub(r"/\*.*?\*/", "", open(h).read(), flags=re.S)
        names |= set(re.findall(r"\b(elsaa_\w+)\s*\(", src))
    return names


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert {"elsaa_forward", "elsaa_workspace_size", "elsaa_last_error",
            "elsaa_check_status", "elsaa_abi_version"} <= names
    for n in names:
        assert hasattr(lib, n), n
    assert set(elsaa.SYMBOLS) <= names


def test_params_struct_matches_header():
    src = open(os.path.join(ROOT, "include", "elsaa.h")).read()
    body = src[src.index("typedef struct elsaa_params"):]
    body = body[body.index("{") + 1:body.index("} elsaa_params;")]
    body = re.sub(r"/\*.*?\*/", "", body, flags=re.S)
    fields = []
    for decl in body.split(";"):
        decl = decl.strip()
        if not decl:
            continue
        typ, rest = decl.split(None, 1)
        for name in rest.split(","):
            fields.append((typ, name.strip()))
    ct = {"int": ctypes.c_int, "float": ctypes.c_float}
    assert len(fields) == len(elsaa.elsaa_params._fields_)
    for (typ, name), (pname, ptype) in zip(fields,
                                           elsaa.elsaa_params._fields_):
        assert ct[typ] is ptype
        assert name == pname or (name == "lambda" and pname == "lam")


def test_abi_version(lib):
    assert elsaa.elsaa_abi_version() == 6


@pytest.mark.parametrize("name", sorted(WORKLOADS))
def test_workspace_size_is_positive_and_deterministic(lib, name):
    p = elsaa.params_for(WORKLOADS[name])
    a = elsaa.elsaa_workspace_size(p)
    assert a > 0 and a % 256 == 0
    assert a == elsaa.elsaa_workspace_size(p)


BAD = [
    (dict(N=1000, block_size=64), elsaa.ELSAA_ERR_INVALID_ARG, "multiple"),
    (dict(causal=2), elsaa.ELSAA_ERR_INVALID_ARG, "causal"),
    (dict(causal=1, dtype="fp32"), elsaa.ELSAA_ERR_UNSUPPORTED, "causal"),
    (dict(causal=1, causal_base_len=0), elsaa.ELSAA_ERR_INVALID_ARG,
     "causal_base_len"),
    (dict(causal=1, causal_chunk=0), elsaa.ELSAA_ERR_INVALID_ARG,
     "causal_chunk"),
    (dict(causal=1, N=192, causal_base_len=2), elsaa.ELSAA_ERR_UNSUPPORTED,
     "odd"),
    (dict(causal=1, N=384, causal_base_len=100), elsaa.ELSAA_ERR_UNSUPPORTED,
     "multiple of 128"),
    (dict(causal=1, neighbor_blocks=1), elsaa.ELSAA_ERR_UNSUPPORTED,
     "neighbor_blocks"),
    (dict(d_h=96), elsaa.ELSAA_ERR_UNSUPPORTED, "d_h"),
    (dict(eps=0.0), elsaa.ELSAA_ERR_INVALID_ARG, "eps"),
    (dict(lam=-1.0), elsaa.ELSAA_ERR_INVALID_ARG, "lambda"),
    (dict(beta=float("nan")), elsaa.ELSAA_ERR_INVALID_ARG, "beta"),
    (dict(block_size=48, N=96), elsaa.ELSAA_ERR_UNSUPPORTED, "block_size"),
    (dict(sort_bits=12), elsaa.ELSAA_ERR_UNSUPPORTED, "sort_bits"),
    (dict(sort_bits=-1), elsaa.ELSAA_ERR_INVALID_ARG, "sort_bits"),
    (dict(race_bits=0), elsaa.ELSAA_ERR_INVALID_ARG, "race_bits"),
    (dict(race_tables=64, race_bits=5), elsaa.ELSAA_ERR_UNSUPPORTED, "1024"),
    (dict(fusion_mode=3), elsaa.ELSAA_ERR_INVALID_ARG, "fusion_mode"),
    (dict(B=0), elsaa.ELSAA_ERR_INVALID_ARG, "positive"),
    (dict(neighbor_blocks=-1), elsaa.ELSAA_ERR_INVALID_ARG, "neighbor"),
    (dict(out_fp32=2), elsaa.ELSAA_ERR_INVALID_ARG, "out_fp32"),
    (dict(selector=2), elsaa.ELSAA_ERR_INVALID_ARG, "selector"),
    (dict(selector=1, topk=8, topk_blocks=0), elsaa.ELSAA_ERR_INVALID_ARG,
     "topk_blocks"),
    (dict(selector=1, topk=8, topk_blocks=5), elsaa.ELSAA_ERR_INVALID_ARG,
     "topk_blocks"),
    (dict(selector=1, topk=129, topk_blocks=2), elsaa.ELSAA_ERR_INVALID_ARG,
     "topk"),
    (dict(selector=1, topk=0, topk_blocks=2), elsaa.ELSAA_ERR_INVALID_ARG,
     "topk"),
    (dict(selector=1, topk=8, topk_blocks=2, neighbor_blocks=1),
     elsaa.ELSAA_ERR_INVALID_ARG, "neighbor_blocks"),
    (dict(selector=1, topk=8, topk_blocks=2, causal=1),
     elsaa.ELSAA_ERR_UNSUPPORTED, "causal"),
    (dict(selector=1, topk=8, topk_blocks=9, N=1024),
     elsaa.ELSAA_ERR_UNSUPPORTED, "512"),
]


def test_selector_workspace_grows_and_backward_refuses(lib):
    base = dict(B=1, H=2, N=1024, d_h=64, block_size=64, race_tables=4)
    a = elsaa.elsaa_workspace_size(elsaa.make_params(**base))
    p = elsaa.make_params(selector=1, topk=64, topk_blocks=2, **base)
    assert elsaa.elsaa_workspace_size(p) > a
    n = ctypes.c_size_t(0)
    rc = lib.elsaa_backward_workspace_size(ctypes.byref(p), ctypes.byref(n))
    assert rc == elsaa.ELSAA_ERR_UNSUPPORTED
    assert "selector" in elsaa.elsaa_last_error()


@pytest.mark.parametrize("N,N0,levels", [(16384, 4096, 2), (1024, 256, 2),
                                         (2048, 300, 3), (512, 4096, 0)])
def test_causal_levels(lib, N, N0, levels):
    p = elsaa.make_params(B=1, H=2, N=N, d_h=128, block_size=128,
                          race_tables=16, causal=1, causal_base_len=N0)
    assert elsaa.elsaa_causal_levels(p) == levels


def test_causal_index_lists_rejects_non_causal(lib):
    p = elsaa.make_params(B=1, H=2, N=256, d_h=64, block_size=64,
                          race_tables=4)
    rc = lib.elsaa_causal_index_lists(ctypes.byref(p), None, 0, None, None)
    assert rc == elsaa.ELSAA_ERR_INVALID_ARG
    assert "causal" in elsaa.elsaa_last_error()


@pytest.mark.parametrize("over,code,word", BAD)
def test_invalid_parameters_rejected(lib, over, code, word):
    kw = dict(B=1, H=2, N=256, d_h=64, block_size=64, race_tables=4)
    kw.update(over)
    p = elsaa.make_params(**kw)
    n = ctypes.c_size_t(0)
    rc = lib.elsaa_workspace_size(ctypes.byref(p), ctypes.byref(n))
    assert rc == code
    assert word in elsaa.elsaa_last_error()


def test_forward_rejects_null_and_small_workspace_before_launch(lib):
    p = elsaa.make_params(B=1, H=1, N=256, d_h=64, block_size=64,
                          race_tables=4)
    fake = 1 << 20  # never dereferenced: validation fails first
    args = [fake] * 5 + [None, None, fake, None, None, None, None, None]
    rc = lib.elsaa_forward(ctypes.byref(p), *args, None, 0, None)
    assert rc == elsaa.ELSAA_ERR_WORKSPACE
    rc = lib.elsaa_forward(ctypes.byref(p), *args, fake, 256, None)
    assert rc == elsaa.ELSAA_ERR_WORKSPACE
    assert "too small" in elsaa.elsaa_last_error()
    args_null = [None] + args[1:]
    rc = lib.elsaa_forward(ctypes.byref(p), *args_null, fake, 1 << 40, None)
    assert rc == elsaa.ELSAA_ERR_INVALID_ARG
    p2 = elsaa.make_params(B=1, H=1, N=256, d_h=64, block_size=64,
                           race_tables=4, dtype="fp32")
    odd = [fake + 2] + args[1:]
    rc = lib.elsaa_forward(ctypes.byref(p2), *odd, fake, 1 << 40, None)
    assert rc == elsaa.ELSAA_ERR_INVALID_ARG
    assert "aligned" in elsaa.elsaa_last_error()
    # element-aligned but not 16-byte aligned (q, then w_race)
    for pos in (0, 4):
        odd = list(args)
        odd[pos] = fake + 8
        rc = lib.elsaa_forward(ctypes.byref(p), *odd, fake, 1 << 40, None)
        assert rc == elsaa.ELSAA_ERR_INVALID_ARG
        assert "16-byte" in elsaa.elsaa_last_error()


def test_missing_library_fails_loudly(tmp_path):
    saved = elsaa._lib
    elsaa._lib = None
    try:
        with pytest.raises(RuntimeError, match="not built"):
            elsaa.load_library(str(tmp_path / "absent.so"))
    finally:
        elsaa._lib = saved


def test_gate_mlp_struct_matches_header():
    src = open(os.path.join(ROOT, "include", "elsaa.h")).read()
    body = src[src.index("typedef struct elsaa_gate_mlp"):]
    body = body[body.index("{") + 1:body.index("} elsaa_gate_mlp;")]
    body = re.sub(r"/\*.*?\*/", "", body, flags=re.S)
    names = [re.findall(r"(\w+)\s*$", d.strip())[0]
             for d in body.split(";") if d.strip()]
    assert names == [f[0] for f in elsaa.elsaa_gate_mlp._fields_]


def test_gates_validation_before_launch(lib):
    p = elsaa.make_params(B=1, H=2, N=256, d_h=64, block_size=64,
                          race_tables=4)
    fake = 1 << 20  # never dereferenced: validation fails first
    m = elsaa.elsaa_gate_mlp(64, fake, fake, fake, fake, None, None, None,
                             1e-6)
    n = ctypes.c_size_t(0)
    assert lib.elsaa_gates_workspace_size(ctypes.byref(p), ctypes.byref(m),
                                          ctypes.byref(n)) == elsaa.ELSAA_OK
    # the bf16 image of [W1; w_lambda; 0] per head after the status word
    assert n.value == 256 + 2 * (64 + 16) * 64 * 2
    for hidden, code in ((24, elsaa.ELSAA_ERR_UNSUPPORTED),
                         (256, elsaa.ELSAA_ERR_UNSUPPORTED),
                         (0, elsaa.ELSAA_ERR_UNSUPPORTED)):
        bad = elsaa.elsaa_gate_mlp(hidden, fake, fake, fake, fake, None,
                                   None, None, 1e-6)
        assert lib.elsaa_gates_workspace_size(
            ctypes.byref(p), ctypes.byref(bad), ctypes.byref(n)) == code
        assert "hidden" in elsaa.elsaa_last_error()
    # lambda requested without its coefficient arrays / floor
    bad = elsaa.elsaa_gate_mlp(64, fake, fake, fake, fake, fake, None, None,
                               1e-6)
    assert lib.elsaa_gates(ctypes.byref(p), ctypes.byref(bad), fake, fake,
                           fake, fake, 1 << 30, None) == \
        elsaa.ELSAA_ERR_INVALID_ARG
    bad = elsaa.elsaa_gate_mlp(64, fake, fake, fake, fake, fake, fake, fake,
                               0.0)
    assert lib.elsaa_gates(ctypes.byref(p), ctypes.byref(bad), fake, fake,
                           fake, fake, 1 << 30, None) == \
        elsaa.ELSAA_ERR_INVALID_ARG
    assert "lambda_min" in elsaa.elsaa_last_error()
    # lambda output missing, workspace too small, misaligned q
    lm = elsaa.elsaa_gate_mlp(64, fake, fake, fake, fake, fake, fake, fake,
                              1e-6)
    assert lib.elsaa_gates(ctypes.byref(p), ctypes.byref(lm), fake, fake,
                           None, fake, 1 << 30, None) == \
        elsaa.ELSAA_ERR_INVALID_ARG
    assert lib.elsaa_gates(ctypes.byref(p), ctypes.byref(m), fake, fake,
                           None, fake, 256, None) == elsaa.ELSAA_ERR_WORKSPACE
    assert lib.elsaa_gates(ctypes.byref(p), ctypes.byref(m), fake + 8, fake,
                           None, fake, 1 << 30, None) == \
        elsaa.ELSAA_ERR_INVALID_ARG
    assert "16-byte" in elsaa.elsaa_last_error()


def test_selftest_arguments_checked_before_launch(lib):
    fake = 1 << 20  # never dereferenced: validation fails first
    assert lib.elsaa_selftest_wait_timeout(None, 256, 100, None) == \
        elsaa.ELSAA_ERR_WORKSPACE
    assert lib.elsaa_selftest_wait_timeout(fake + 16, 256, 100, None) == \
        elsaa.ELSAA_ERR_WORKSPACE
    for bad in (0, 5000):
        assert lib.elsaa_selftest_wait_timeout(fake, 256, bad, None) == \
            elsaa.ELSAA_ERR_INVALID_ARG
        assert "limit_ms" in elsaa.elsaa_last_error()
