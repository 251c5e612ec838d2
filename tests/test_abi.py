"""The C-ABI library builds, loads and exports every symbol include/treeflash.h declares; host-side
argument validation works without a GPU (no compute call is made here)."""
import ctypes
import os
import re

import pytest

import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2606_03819_gb300 import binding
    if not os.path.exists(binding.LIB_PATH):
        from paper_2606_03819_gb300 import build
        build.build()
    return binding.load_library()


def declared_functions():
    src = open(os.path.join(ROOT, "include", "treeflash.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(tf_[a-z0-9_]+)\s*\(", src)))


def test_header_declares_the_four_calls_of_the_path():
    names = declared_functions()
    for n in ("tf_stage1_marginals", "tf_stage2_ar_approx", "tf_build_tree", "tf_tree_mask"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    from paper_2606_03819_gb300 import binding
    names = declared_functions()
    assert set(names) == set(binding.EXPORTS)
    for n in names:
        assert hasattr(lib, n), n


def test_version_and_status_strings(lib):
    assert lib.tf_version() >= 100
    for s in range(7):
        assert lib.tf_status_string(s)


def _dims(**kw):
    from paper_2606_03819_gb300.binding import Dims
    base = dict(batch=1, d=128, V=2048, I=512, gamma=4, M=4, K2=12, B=12, dtype="f32", mode="ar")
    base.update(kw)
    return Dims(**base)


def test_workspace_size_and_validation(lib):
    from paper_2606_03819_gb300 import binding as Bn
    assert Bn.tf_workspace_size(_dims()) > 0
    q8 = Bn.Dims.from_config(synth.get_config("q8_b64"))
    n = Bn.tf_workspace_size(q8)
    # partials of the larger pass: 241 rows x 594 blocks x 72 bytes, plus h', X, A
    assert n >= 241 * 594 * 72 + 241 * 4096 * 2 * 4
    bad = [dict(batch=0), dict(V=8, K2=12), dict(gamma=0), dict(M=0), dict(temperature=0.0),
           dict(mode="nope"), dict(I=0)]
    for kw in bad:
        if kw.get("mode") == "nope":
            continue
        with pytest.raises(Bn.TreeFlashError) as e:
            Bn.tf_workspace_size(_dims(**kw))
        assert e.value.status == Bn.TF_ERR_INVALID_ARG, kw
    for kw in (dict(M=65), dict(K2=513, V=4096), dict(B=2000), dict(gamma=65), dict(dtype="bf16", d=100),
               dict(dtype="bf16", I=100)):
        with pytest.raises(Bn.TreeFlashError) as e:
            Bn.tf_workspace_size(_dims(**kw))
        assert e.value.status == Bn.TF_ERR_UNSUPPORTED, kw


def test_null_arguments_are_rejected_before_any_gpu_work(lib):
    from paper_2606_03819_gb300 import binding as Bn
    d = _dims()
    c = d.c()
    w = Bn.TfWeights()
    # null workspace -> TF_ERR_WORKSPACE; null dims -> TF_ERR_INVALID_ARG; all host-side
    assert lib.tf_stage1_marginals(None, ctypes.byref(w), None, None, None, None, 0, None) == Bn.TF_ERR_INVALID_ARG
    assert lib.tf_stage1_marginals(ctypes.byref(c), ctypes.byref(w), None, None, None, None, 0,
                                   None) == Bn.TF_ERR_WORKSPACE
    assert lib.tf_build_tree(ctypes.byref(c), *([None] * 10), None) == Bn.TF_ERR_INVALID_ARG
    assert lib.tf_tree_mask(ctypes.byref(c), None, None, None, None, None, None) == Bn.TF_ERR_INVALID_ARG
    assert lib.tf_status_reset(None, 0, None) == Bn.TF_ERR_WORKSPACE
    flags = ctypes.c_int32()
    assert lib.tf_status_read(None, 0, ctypes.byref(flags), None) == Bn.TF_ERR_WORKSPACE
    n = ctypes.c_size_t()
    assert lib.tf_workspace_size(ctypes.byref(c), None) == Bn.TF_ERR_INVALID_ARG


def test_product_path_never_imports_the_oracle():
    # the binding and package sources must not reference oracle/ (no CPU fallback)
    pkg = os.path.join(ROOT, "paper_2606_03819_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h", ".cpp")):
                txt = open(os.path.join(dirpath, f)).read()
                assert "oracle" not in txt.lower(), f


def _header_arity():
    src = open(os.path.join(ROOT, "include", "treeflash.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    out = {}
    for m in re.finditer(r"\b(tf_[a-z0-9_]+)\s*\(([^)]*)\)\s*;", src):
        args = m.group(2).strip()
        out[m.group(1)] = 0 if args in ("", "void") else args.count(",") + 1
    return out


def test_binding_signatures_match_header_arity(lib):
    arity = _header_arity()
    assert set(arity) == set(declared_functions())
    for name, n in arity.items():
        assert len(getattr(lib, name).argtypes) == n, name


def _header_struct_fields(name):
    src = open(os.path.join(ROOT, "include", "treeflash.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    body = re.search(r"typedef struct \{([^}]*)\}\s*" + name + r"\s*;", src).group(1)
    return re.findall(r"(\w+)\s*;", body)


def test_binding_structs_match_header_layout():
    # the ctypes structs must list the header's fields in the header's order (the struct is
    # passed by pointer, so a missing or reordered field would shift every later one)
    from paper_2606_03819_gb300 import binding as Bn
    assert [f for f, _ in Bn.TfDims._fields_] == _header_struct_fields("tf_dims")
    assert [f for f, _ in Bn.TfWeights._fields_] == _header_struct_fields("tf_weights")
    assert ctypes.sizeof(Bn.TfDims) == 4 * len(Bn.TfDims._fields_)


def test_approximator_kind_validation(lib):
    from paper_2606_03819_gb300 import binding as Bn
    # the linear approximator has no intermediate width: I is ignored, also its bf16 alignment
    assert Bn.tf_workspace_size(_dims(approx="linear", I=0)) > 0
    assert Bn.tf_workspace_size(_dims(approx="linear", I=100, dtype="bf16")) > 0
    # it needs no A buffer, so its workspace is smaller than the SwiGLU one of the same shape
    assert Bn.tf_workspace_size(_dims(approx="linear")) < Bn.tf_workspace_size(_dims())
    # an unknown kind is rejected in TreeFlash mode and ignored by the marginal modes
    c = _dims().c()
    c.approx = 7
    n = ctypes.c_size_t()
    assert lib.tf_workspace_size(ctypes.byref(c), ctypes.byref(n)) == Bn.TF_ERR_INVALID_ARG
    c.mode = Bn.MODES["marginal"]
    assert lib.tf_workspace_size(ctypes.byref(c), ctypes.byref(n)) == Bn.TF_OK


def test_linear_approximator_needs_w_lin_not_the_swiglu_weights(lib):
    # host-side weight checks run before any GPU work: a null w_lin is rejected for the linear
    # approximator, null SwiGLU weights for the SwiGLU one (argument order: dims, weights,
    # hidden, root_tok, top_ids, h_prime, ws, ws_bytes, stream)
    from paper_2606_03819_gb300 import binding as Bn
    buf = ctypes.create_string_buffer(1 << 16)
    fake = ctypes.addressof(buf) + (-ctypes.addressof(buf)) % 256   # aligned, never dereferenced
    for approx, missing in (("linear", "w_lin"), ("swiglu", "w_down")):
        d = _dims(approx=approx)
        c = d.c()
        w = Bn.TfWeights(*[None if k == missing else fake for k in Bn.WEIGHT_KEYS])
        ws_bytes = Bn.tf_workspace_size(d)
        st = lib.tf_ar_approx(ctypes.byref(c), ctypes.byref(w), fake, fake, fake, None, fake, ws_bytes, None)
        assert st == Bn.TF_ERR_INVALID_ARG, approx


def test_two_prev_approximator_layout(lib):
    # two previous tokens: 1 + M + M^2 (gamma - 2) stage-2 rows of width 3d, and room for a residual
    # row per stage-2 row; the row count shows in the views (no GPU work: host-side layout only)
    from paper_2606_03819_gb300 import binding as Bn
    d1 = _dims()
    d2 = _dims(approx="swiglu_2prev")
    assert d2.R == 1 + 4 + 16 * 2 == 37 and d1.R == 13
    n2 = Bn.tf_workspace_size(d2)
    assert n2 > Bn.tf_workspace_size(d1)
    buf = ctypes.create_string_buffer(n2 + 256)
    ws = ctypes.addressof(buf) + (-ctypes.addressof(buf)) % 256
    p, nb = ctypes.c_void_p(), ctypes.c_size_t()
    c = d2.c()
    assert lib.tf_workspace_view(ctypes.byref(c), ws, n2, Bn.TF_VIEW_X, ctypes.byref(p), ctypes.byref(nb)) == 0
    assert nb.value == 37 * 3 * 128 * 4
    assert lib.tf_workspace_view(ctypes.byref(c), ws, n2, Bn.TF_VIEW_H_PRIME, ctypes.byref(p),
                                 ctypes.byref(nb)) == 0
    assert nb.value == 37 * 128 * 4
    # gamma = 1 leaves one row; the marginal modes ignore the approximator kind
    assert _dims(approx="swiglu_2prev", gamma=1).R == 1
    assert Bn.tf_workspace_size(_dims(approx="swiglu_2prev", mode="marginal")) == \
        Bn.tf_workspace_size(_dims(mode="marginal"))


def test_view_and_mode_checks_before_any_gpu_work(lib):
    # host-only checks: the SwiGLU intermediate view is empty for the linear approximator; the
    # approximator calls need TreeFlash mode; the merge's k is bounded by 512 and V
    from paper_2606_03819_gb300 import binding as Bn
    d = _dims(approx="linear")
    n = Bn.tf_workspace_size(d)
    buf = ctypes.create_string_buffer(n + 256)
    ws = ctypes.addressof(buf) + (-ctypes.addressof(buf)) % 256
    p, nb = ctypes.c_void_p(), ctypes.c_size_t()
    c = d.c()
    assert lib.tf_workspace_view(ctypes.byref(c), ws, n, Bn.TF_VIEW_A, ctypes.byref(p), ctypes.byref(nb)) == 0
    assert nb.value == 0
    assert lib.tf_workspace_view(ctypes.byref(c), ws, n, 99, ctypes.byref(p), ctypes.byref(nb)) == \
        Bn.TF_ERR_INVALID_ARG
    marg = _dims(mode="marginal")
    cm = marg.c()
    nm = Bn.tf_workspace_size(marg)
    w = Bn.TfWeights(*[ws for _ in Bn.WEIGHT_KEYS])
    assert lib.tf_ar_approx(ctypes.byref(cm), ctypes.byref(w), ws, ws, ws, None, ws, nm, None) == \
        Bn.TF_ERR_INVALID_ARG
    assert lib.tf_workspace_h_prime(ctypes.byref(cm), ws, nm, ctypes.byref(p)) == Bn.TF_ERR_INVALID_ARG
    assert lib.tf_workspace_view(ctypes.byref(cm), ws, nm, Bn.TF_VIEW_X, ctypes.byref(p),
                                 ctypes.byref(nb)) == Bn.TF_ERR_INVALID_ARG
    # a workspace one byte short, or misaligned, is refused
    assert lib.tf_workspace_view(ctypes.byref(c), ws, n - 1, Bn.TF_VIEW_X, ctypes.byref(p),
                                 ctypes.byref(nb)) == Bn.TF_ERR_WORKSPACE
    assert lib.tf_workspace_view(ctypes.byref(c), ws + 16, n, Bn.TF_VIEW_X, ctypes.byref(p),
                                 ctypes.byref(nb)) == Bn.TF_ERR_WORKSPACE
