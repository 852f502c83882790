"""The C ABI on the CPU: the library loads, exports every function
include/ember.h declares, and rejects bad arguments on the host before
anything reaches a GPU.  No compute call is made here."""
import ctypes
import json
import os
import re

import pytest

from paper_2607_01455_gb300 import ember as E
from paper_2607_01455_gb300.build import INCLUDE, build_library

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built():
    build_library()


def header_functions():
    text = open(os.path.join(INCLUDE, "ember.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return set(re.findall(r"\b(ember_[a-z_]+)\s*\(", text))


def test_library_exports_every_declared_function():
    declared = header_functions()
    assert declared == set(E.EXPORTS)
    lib = ctypes.CDLL(E.LIB_PATH)
    for name in declared:
        assert hasattr(lib, name), name
    assert E.ember_abi_version() == 2


def test_status_strings():
    for code in range(0, 9):
        assert E.ember_status_string(code)
    assert E.ember_status_string(0) == "ok"
    assert E.ember_status_string(99) == "unknown status"


def test_defaults_follow_algorithm_1():
    hp = E.ember_hparams_default()
    assert (hp.beta2, hp.eps, hp.maximize, hp.bias_correction, hp.variant) == (0.999, 1e-8, 0, 1, 0)


@pytest.mark.parametrize("V,D", [(1, 1), (1024, 64), (151936, 896), (128256, 8192), (5, 2047)])
def test_state_is_exactly_v_plus_d(V, D):
    h = E.ember_create(V, D)
    try:
        assert E.ember_state_numel(h) == V + D
        assert E.ember_workspace_bytes(h, 0) > 0
        assert E.ember_workspace_bytes(h, 1000) > E.ember_workspace_bytes(h, 0)
        assert E.ember_workspace_bytes(h, -1) == 0
    finally:
        E.ember_destroy(h)


def test_paper_state_sizes_through_the_library():
    """Ember's printed state sizes (Section 3.1 table, Sections 4 and 5.1)
    follow from ember_state_numel * 4 bytes per table."""
    with open(os.path.join(ROOT, "tests", "golden", "state_sizes.json")) as f:
        entries = json.load(f)["entries"]
    div = {"KiB": 1024, "MiB": 1024 ** 2}
    for e in entries:
        h = E.ember_create(e["V"], e["D"])
        try:
            nbytes = e["tables"] * 4 * E.ember_state_numel(h)
        finally:
            E.ember_destroy(h)
        val, unit = e["ember"][0], e["ember"][1]
        tol = 0.05 if "approx" in e["ember"] else 0.005
        assert nbytes / div[unit] == pytest.approx(val, rel=tol), e["model"]


@pytest.mark.parametrize("kw,status", [
    (dict(V=0, D=4), E.EMBER_ERR_INVALID_ARG),
    (dict(V=4, D=0), E.EMBER_ERR_INVALID_ARG),
    (dict(V=-3, D=4), E.EMBER_ERR_INVALID_ARG),
    (dict(V=1 << 40, D=1 << 30), E.EMBER_ERR_INVALID_ARG),
    (dict(V=4, D=4, wdtype=7), E.EMBER_ERR_DTYPE),
    (dict(V=4, D=4, beta2=1.0), E.EMBER_ERR_INVALID_ARG),
    (dict(V=4, D=4, beta2=-0.1), E.EMBER_ERR_INVALID_ARG),
    (dict(V=4, D=4, eps=-1.0), E.EMBER_ERR_INVALID_ARG),
    (dict(V=4, D=4, eps=float("inf")), E.EMBER_ERR_INVALID_ARG),
    (dict(V=4, D=4, variant=3), E.EMBER_ERR_INVALID_ARG),
    (dict(V=4, D=4, maximize=2), E.EMBER_ERR_INVALID_ARG),
    (dict(V=4, D=65537), E.EMBER_ERR_UNSUPPORTED),
    (dict(V=4, D=1 << 20), E.EMBER_ERR_UNSUPPORTED),
    (dict(V=1 << 31, D=4), E.EMBER_ERR_UNSUPPORTED),
])
def test_create_rejects(kw, status):
    hp = E.ember_hparams_default()
    for k in ("beta2", "eps", "variant", "maximize"):
        if k in kw:
            setattr(hp, k, kw.pop(k))
    with pytest.raises(E.EmberError) as ex:
        E.ember_create(kw["V"], kw["D"], hp, kw.get("wdtype", E.EMBER_BF16))
    assert ex.value.status == status


def test_from_host_refuses_row_only_variant():
    hp = E.ember_hparams_default()
    hp.variant = E.EMBER_VARIANT_ROW
    h = E.ember_create(16, 8, hp)
    try:
        fake = 1 << 20
        assert E.lib().ember_step_dense_from_host(h, fake, fake, fake, fake, 1e-3, 1, None) == \
            E.EMBER_ERR_UNSUPPORTED
    finally:
        E.ember_destroy(h)


@pytest.mark.parametrize("V,D", [(12, 16), (16, 12), (1001, 8)])
def test_lmhead_needs_multiples_of_8(V, D):
    h = E.ember_create(V, D)
    try:
        fake = 1 << 20
        assert E.lib().ember_lmhead_grad(h, fake, fake, 4, fake, None) == E.EMBER_ERR_UNSUPPORTED
        assert E.lib().ember_step_lmhead(h, fake, fake, fake, 4, fake, fake, 1e-3, 1, None) == \
            E.EMBER_ERR_UNSUPPORTED
    finally:
        E.ember_destroy(h)


def test_create_accepts_limits():
    # widths past one CTA's row (8192, or 2048 without 16-byte vectors) run
    # in column panels, up to 65536
    for V, D in [(1, 8192), (3, 2048), (2, 2047), (1, 3), (2, 8196), (2, 2049), (1, 65536), (1, 65533)]:
        E.ember_destroy(E.ember_create(V, D))


def test_step_and_bind_reject_on_host():
    lib = E.lib()
    h = E.ember_create(16, 8)
    try:
        fake = 1 << 20  # never dereferenced: every call below fails its checks first
        # workspace: null, misaligned, too small
        assert lib.ember_bind_workspace(h, None, 1 << 20, 0, None) == E.EMBER_ERR_INVALID_ARG
        assert lib.ember_bind_workspace(h, fake + 8, 1 << 20, 0, None) == E.EMBER_ERR_ALIGNMENT
        assert lib.ember_bind_workspace(h, fake, 16, 0, None) == E.EMBER_ERR_WORKSPACE
        assert lib.ember_bind_workspace(h, fake, 1 << 20, -1, None) == E.EMBER_ERR_INVALID_ARG
        assert lib.ember_bind_workspace(None, fake, 1 << 20, 0, None) == E.EMBER_ERR_INVALID_ARG
        # dense step: nulls, t < 1, non-finite lr, misaligned, no workspace bound
        assert lib.ember_step_dense(h, None, fake, fake, 1e-3, 1, None) == E.EMBER_ERR_INVALID_ARG
        assert lib.ember_step_dense(h, fake, None, fake, 1e-3, 1, None) == E.EMBER_ERR_INVALID_ARG
        assert lib.ember_step_dense(h, fake, fake, None, 1e-3, 1, None) == E.EMBER_ERR_INVALID_ARG
        assert lib.ember_step_dense(h, fake, fake, fake, 1e-3, 0, None) == E.EMBER_ERR_INVALID_ARG
        assert lib.ember_step_dense(h, fake, fake, fake, float("nan"), 1, None) == E.EMBER_ERR_INVALID_ARG
        assert lib.ember_step_dense(h, fake + 1, fake, fake, 1e-3, 1, None) == E.EMBER_ERR_ALIGNMENT
        assert lib.ember_step_dense(h, fake, fake + 2, fake, 1e-3, 1, None) == E.EMBER_ERR_ALIGNMENT
        assert lib.ember_step_dense(h, fake, fake, fake, 1e-3, 1, None) == E.EMBER_ERR_WORKSPACE
        assert lib.ember_step_dense(None, fake, fake, fake, 1e-3, 1, None) == E.EMBER_ERR_INVALID_ARG
        # sparse step
        assert lib.ember_step_sparse(h, fake, fake, 0, -1, fake, fake, 1e-3, 1, None) == E.EMBER_ERR_INVALID_ARG
        assert lib.ember_step_sparse(h, fake, None, 0, 4, fake, fake, 1e-3, 1, None) == E.EMBER_ERR_INVALID_ARG
        assert lib.ember_step_sparse(h, fake, fake, 5, 4, fake, fake, 1e-3, 1, None) == E.EMBER_ERR_DTYPE
        assert lib.ember_step_sparse(h, fake, fake, 1, 4, fake, fake, 1e-3, 0, None) == E.EMBER_ERR_INVALID_ARG
        # dense step from host memory: rejected before any CUDA call
        fh = lib.ember_step_dense_from_host
        assert fh(h, fake, None, fake, fake, 1e-3, 1, None) == E.EMBER_ERR_INVALID_ARG
        assert fh(h, fake, fake, None, fake, 1e-3, 1, None) == E.EMBER_ERR_INVALID_ARG
        assert fh(h, fake, fake, fake, fake, 1e-3, 0, None) == E.EMBER_ERR_INVALID_ARG
        assert fh(h, fake, fake + 2, fake, fake, 1e-3, 1, None) == E.EMBER_ERR_ALIGNMENT
        assert fh(h, fake, fake, fake, fake, 1e-3, 1, None) == E.EMBER_ERR_WORKSPACE
        # LM-head gradient and fused step: rejected before any CUDA call
        lg, sl = lib.ember_lmhead_grad, lib.ember_step_lmhead
        assert lg(h, None, fake, 4, fake, None) == E.EMBER_ERR_INVALID_ARG
        assert lg(h, fake, fake, 0, fake, None) == E.EMBER_ERR_INVALID_ARG
        assert lg(h, fake, fake, 1 << 31, fake, None) == E.EMBER_ERR_INVALID_ARG
        assert lg(h, fake + 8, fake, 4, fake, None) == E.EMBER_ERR_ALIGNMENT
        assert lg(h, fake, fake, 4, fake + 4, None) == E.EMBER_ERR_ALIGNMENT
        assert lg(h, fake, fake, 4, fake, None) == E.EMBER_ERR_WORKSPACE
        assert sl(h, fake, fake, fake, 4, fake, fake, 1e-3, 0, None) == E.EMBER_ERR_INVALID_ARG
        assert sl(h, None, fake, fake, 4, fake, fake, 1e-3, 1, None) == E.EMBER_ERR_INVALID_ARG
        assert sl(h, fake, fake, fake, 4, fake, fake, float("inf"), 1, None) == E.EMBER_ERR_INVALID_ARG
        assert sl(h, fake, fake, fake, 4, fake, fake, 1e-3, 1, None) == E.EMBER_ERR_WORKSPACE
        assert E.lib().ember_get_device_status(h, None) == E.EMBER_ERR_WORKSPACE
        assert lib.ember_get_device_status(None, None) == E.EMBER_ERR_INVALID_ARG
    finally:
        E.ember_destroy(h)
    E.ember_destroy(0)  # NULL is ignored


@pytest.mark.parametrize("D", [1, 7, 2047, 2048, 2049, 3001, 4096, 8192, 8196, 10001, 12288, 16384,
                               24576, 65533, 65536])
def test_column_panels_follow_the_cta_row_width(D):
    """A CTA holds 8192 columns of a row on the 16-byte path (D % 4 == 0),
    2048 on the scalar one; a wider table runs in the fewest panels that
    fit, ceil(D / width)."""
    h = E.ember_create(3, D)
    try:
        vec = E.ember_column_panels(h, True)
        sca = E.ember_column_panels(h, False)
        assert sca == -(-D // 2048)
        assert vec == (-(-D // 8192) if D % 4 == 0 else sca)
    finally:
        E.ember_destroy(h)
    assert E.lib().ember_column_panels(None, 1) == 0
