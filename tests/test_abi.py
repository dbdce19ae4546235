"""The C ABI without a GPU: the libraries load, export every function that
include/*.h declares, and reject bad arguments on the host before any launch."""
import ctypes
import math
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2608_02625_gb300")


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2608_02625_gb300 import build
    build.build()


def declared_functions(header):
    text = open(os.path.join(ROOT, "include", header)).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[\w\*\s]+?\b(dlm_\w+)\s*\(", text, flags=re.M)))


@pytest.mark.parametrize("header,lib", [("dlmrefine.h", "libdlmrefine.so"), ("dlmsynth.h", "libdlmsynth.so")])
def test_exports_every_declared_symbol(header, lib):
    names = declared_functions(header)
    assert len(names) >= 2
    so = ctypes.CDLL(os.path.join(PKG, lib))
    for n in names:
        assert hasattr(so, n), f"{lib} does not export {n}"


def test_version_and_status_strings():
    from paper_2608_02625_gb300 import binding as B
    assert B.dlm_version() == 201
    assert B.dlm_status_string(0) == "ok"
    assert "dtype" in B.dlm_status_string(-2)


# ---- host-side validation: fake device pointers are never dereferenced

def T(dtype, shape, ptr=0x100000, strides=None):
    from paper_2608_02625_gb300.binding import DlmTensor
    d = DlmTensor()
    d.data = ptr
    d.dtype = dtype
    d.ndim = len(shape)
    if strides is None:
        strides, acc = [], 1
        for s in reversed(shape):
            strides.insert(0, acc)
            acc *= s
    for i, (s, st) in enumerate(zip(shape, strides)):
        d.shape[i] = s
        d.stride[i] = st
    return d


BF16, F32, I32, U8 = 1, 2, 3, 4
MB = 1 << 26


def attn(q, k, v, sl, o):
    from paper_2608_02625_gb300.binding import lib
    r = lambda d: ctypes.byref(d) if d is not None else None
    return lib.dlm_bidir_attn(r(q), r(k), r(v), r(sl), r(o))


def good_attn(D=128, dtype=BF16, Hq=8, Hkv=2):
    return (T(dtype, [2, 16, Hq, D], 1 * MB), T(dtype, [2, 16, Hkv, D], 2 * MB), T(dtype, [2, 16, Hkv, D], 3 * MB),
            T(I32, [2], 4 * MB), T(dtype, [2, 16, Hq, D], 5 * MB))


@pytest.mark.parametrize("case,status", [
    ("null_q", -1), ("dtype_mismatch", -2), ("int_dtype", -2), ("head_dim_96", -3), ("gqa_not_multiple", -3),
    ("out_shape", -3), ("seq_lens_shape", -3), ("inner_stride", -4), ("misaligned_bf16", -5),
    ("out_overlaps_q", -6), ("rank3", -3),
])
def test_attn_rejects(case, status):
    q, k, v, sl, o = good_attn()
    if case == "null_q":
        q = None
    elif case == "dtype_mismatch":
        k = T(F32, [2, 16, 2, 128], 2 * MB)
    elif case == "int_dtype":
        q, k, v, sl, o = good_attn(dtype=I32)
    elif case == "head_dim_96":
        q, k, v, sl, o = good_attn(D=96)
    elif case == "gqa_not_multiple":
        q, k, v, sl, o = good_attn(Hq=6, Hkv=4)
    elif case == "out_shape":
        o = T(BF16, [2, 16, 4, 128], 5 * MB)
    elif case == "seq_lens_shape":
        sl = T(I32, [3], 4 * MB)
    elif case == "inner_stride":
        q = T(BF16, [2, 16, 8, 128], 1 * MB, strides=[16 * 8 * 256, 8 * 256, 256, 2])
    elif case == "misaligned_bf16":
        q = T(BF16, [2, 16, 8, 128], 1 * MB + 2)
    elif case == "out_overlaps_q":
        o = T(BF16, [2, 16, 8, 128], 1 * MB + 256)
    elif case == "rank3":
        q = T(BF16, [2, 16, 1024], 1 * MB)
    assert attn(q, k, v, sl, o) == status


def vocab(lg, am, cf, ls):
    from paper_2608_02625_gb300.binding import lib
    return lib.dlm_vocab_confidence(*(ctypes.byref(d) if d is not None else None for d in (lg, am, cf, ls)))


@pytest.mark.parametrize("case,status", [
    ("null_conf", -1), ("logits_int", -2), ("argmax_f32", -2), ("count_mismatch", -3), ("strided_out", -4),
    ("outputs_overlap", -6),
])
def test_vocab_rejects(case, status):
    lg, am, cf, ls = T(BF16, [4, 1000], 1 * MB), T(I32, [4], 2 * MB), T(F32, [4], 3 * MB), T(F32, [4], 4 * MB)
    if case == "null_conf":
        cf = None
    elif case == "logits_int":
        lg = T(I32, [4, 1000], 1 * MB)
    elif case == "argmax_f32":
        am = T(F32, [4], 2 * MB)
    elif case == "count_mismatch":
        cf = T(F32, [5], 3 * MB)
    elif case == "strided_out":
        ls = T(F32, [4], 4 * MB, strides=[2])
    elif case == "outputs_overlap":
        ls = T(F32, [4], 3 * MB + 4)
    assert vocab(lg, am, cf, ls) == status


def update(params, **over):
    from paper_2608_02625_gb300.binding import lib
    d = dict(tok=T(I32, [2, 8], 1 * MB), msk=T(U8, [2, 8], 2 * MB), am=T(I32, [2, 8], 3 * MB),
             cf=T(F32, [2, 8], 4 * MB), nt=T(I32, [2, 8], 5 * MB), nm=T(U8, [2, 8], 6 * MB),
             ne=T(I32, [2], 7 * MB))
    d.update(over)
    r = lambda x: ctypes.byref(x) if x is not None else None
    return lib.dlm_refine_update(r(d["tok"]), r(d["msk"]), r(d["am"]), r(d["cf"]),
                                 ctypes.byref(params) if params is not None else None,
                                 r(d["nt"]), r(d["nm"]), r(d["ne"]))


def P(**kw):
    from paper_2608_02625_gb300.binding import DlmRefineParams
    base = dict(edit_threshold=0.8, remask_k=2, remask_frac=0.0, mask_id=99, prompt_lens=8 * MB, seq_lens=9 * MB)
    base.update(kw)
    return DlmRefineParams(**base)


@pytest.mark.parametrize("case,status", [
    ("null_params", -1), ("nan_threshold", -6), ("frac_above_one", -6), ("frac_nan", -6), ("mask_dtype", -2),
    ("shape_mismatch", -3), ("n_edits_shape", -3), ("partial_alias", -6), ("output_overlaps_input", -6),
    ("null_prompt_lens", -1), ("null_seq_lens", -1), ("misaligned_seq_lens", -5),
])
def test_update_rejects(case, status):
    if case == "null_params":
        assert update(None) == status
    elif case == "nan_threshold":
        assert update(P(edit_threshold=math.nan)) == status
    elif case == "frac_above_one":
        assert update(P(remask_k=-1, remask_frac=1.5)) == status
    elif case == "frac_nan":
        assert update(P(remask_k=-1, remask_frac=math.nan)) == status
    elif case == "mask_dtype":
        assert update(P(), msk=T(I32, [2, 8], 2 * MB)) == status
    elif case == "shape_mismatch":
        assert update(P(), am=T(I32, [2, 9], 3 * MB)) == status
    elif case == "n_edits_shape":
        assert update(P(), ne=T(I32, [3], 7 * MB)) == status
    elif case == "partial_alias":
        assert update(P(), nt=T(I32, [2, 8], 1 * MB + 4)) == status
    elif case == "output_overlaps_input":
        assert update(P(), nt=T(I32, [2, 8], 4 * MB)) == status
    elif case == "null_prompt_lens":
        assert update(P(prompt_lens=None)) == status
    elif case == "null_seq_lens":
        assert update(P(seq_lens=None)) == status
    elif case == "misaligned_seq_lens":
        assert update(P(seq_lens=9 * MB + 2)) == status


def test_last_error_message():
    from paper_2608_02625_gb300.binding import lib
    q, k, v, sl, o = good_attn(D=96)
    assert attn(q, k, v, sl, o) == -3
    assert b"head_dim" in lib.dlm_last_error()


def step(params, ws=10 * MB, ws_bytes=8, **over):
    from paper_2608_02625_gb300.binding import lib
    d = dict(lg=T(BF16, [16, 1000], 11 * MB), tok=T(I32, [2, 8], 1 * MB), msk=T(U8, [2, 8], 2 * MB),
             am=T(I32, [2, 8], 3 * MB), cf=T(F32, [2, 8], 4 * MB), ls=T(F32, [2, 8], 12 * MB),
             nt=T(I32, [2, 8], 5 * MB), nm=T(U8, [2, 8], 6 * MB), ne=T(I32, [2], 7 * MB))
    d.update(over)
    r = lambda x: ctypes.byref(x) if x is not None else None
    return lib.dlm_refine_step(r(d["lg"]), r(d["tok"]), r(d["msk"]), ctypes.byref(params) if params else None,
                               r(d["am"]), r(d["cf"]), r(d["ls"]), r(d["nt"]), r(d["nm"]), r(d["ne"]),
                               ctypes.c_void_p(ws), ctypes.c_size_t(ws_bytes))


def test_step_workspace_bytes():
    from paper_2608_02625_gb300.binding import lib
    assert [lib.dlm_refine_step_workspace_bytes(b) for b in (0, 1, 32, -3)] == [0, 4, 128, 0]


@pytest.mark.parametrize("case,status", [
    ("null_params", -1), ("null_workspace", -1), ("workspace_small", -6), ("workspace_misaligned", -5),
    ("rows_not_BL", -3), ("logits_3d_mismatch", -3), ("strided_conf", -4), ("lse_overlaps_new_tokens", -6),
    ("argmax_overlaps_tokens", -6), ("nan_threshold", -6), ("workspace_overlaps_lse", -6),
])
def test_step_rejects(case, status):
    if case == "null_params":
        assert step(None) == status
    elif case == "null_workspace":
        assert step(P(), ws=0) == status
    elif case == "workspace_small":
        assert step(P(), ws_bytes=7) == status
    elif case == "workspace_misaligned":
        assert step(P(), ws=10 * MB + 2) == status
    elif case == "rows_not_BL":
        assert step(P(), lg=T(BF16, [15, 1000], 11 * MB),
                    am=T(I32, [15], 3 * MB), cf=T(F32, [15], 4 * MB), ls=T(F32, [15], 12 * MB)) == status
    elif case == "logits_3d_mismatch":
        assert step(P(), lg=T(BF16, [4, 4, 1000], 11 * MB)) == status
    elif case == "strided_conf":
        assert step(P(), cf=T(F32, [2, 8], 4 * MB, strides=[16, 1])) == status
    elif case == "lse_overlaps_new_tokens":
        assert step(P(), ls=T(F32, [2, 8], 5 * MB + 8)) == status
    elif case == "argmax_overlaps_tokens":
        assert step(P(), am=T(I32, [2, 8], 1 * MB)) == status
    elif case == "nan_threshold":
        assert step(P(edit_threshold=math.nan)) == status
    elif case == "workspace_overlaps_lse":
        assert step(P(), ws=12 * MB + 60) == status


def test_static_step_rejects_batch_above_maximum_on_the_host():
    from paper_2608_02625_gb300.binding import lib
    B = 4097
    d = dict(lg=T(BF16, [B, 16], 11 * MB), tok=T(I32, [B, 1], 1 * MB), msk=T(U8, [B, 1], 2 * MB),
             am=T(I32, [B, 1], 3 * MB), cf=T(F32, [B, 1], 4 * MB), ls=T(F32, [B, 1], 12 * MB),
             nt=T(I32, [B, 1], 5 * MB), nm=T(U8, [B, 1], 6 * MB), ne=T(I32, [B], 7 * MB))
    r = ctypes.byref
    st = lib.dlm_refine_step_static(r(d["lg"]), r(d["tok"]), r(d["msk"]), r(P()), r(d["am"]), r(d["cf"]),
                                    r(d["ls"]), r(d["nt"]), r(d["nm"]), r(d["ne"]))
    assert st == -3
    assert b"4096" in lib.dlm_last_error()


def test_loop_calls_rejected_on_the_host():
    from paper_2608_02625_gb300.binding import lib
    assert lib.dlm_set_stream(None) == 0
    steps = ctypes.c_void_p(13 * MB)
    assert lib.dlm_loop_begin(steps) == -6                   # legacy default stream cannot be recorded
    assert b"stream" in lib.dlm_last_error()
    h = ctypes.c_void_p()
    assert lib.dlm_loop_end(ctypes.c_void_p(7 * MB), 2, 4, ctypes.byref(h)) == -6   # nothing recorded
    assert lib.dlm_loop_cancel() == 0
    assert lib.dlm_loop_launch(None) == -1
    assert lib.dlm_loop_destroy(None) == 0


@pytest.mark.parametrize("case,status", [
    ("ok_shape_mismatch", -3), ("tokens_f32", -2), ("strided_prob", -4), ("prob_overlaps_lse", -6), ("null_lse", -1),
])
def test_token_prob_rejects(case, status):
    from paper_2608_02625_gb300.binding import lib
    lg, tk, ls, pr = T(BF16, [4, 1000], 1 * MB), T(I32, [4], 2 * MB), T(F32, [4], 3 * MB), T(F32, [4], 4 * MB)
    if case == "ok_shape_mismatch":
        tk = T(I32, [5], 2 * MB)
    elif case == "tokens_f32":
        tk = T(F32, [4], 2 * MB)
    elif case == "strided_prob":
        pr = T(F32, [4], 4 * MB, strides=[2])
    elif case == "prob_overlaps_lse":
        pr = T(F32, [4], 3 * MB + 4)
    elif case == "null_lse":
        ls = None
    r = lambda x: ctypes.byref(x) if x is not None else None
    assert lib.dlm_token_prob(r(lg), r(tk), r(ls), r(pr)) == status


@pytest.mark.parametrize("case,status", [("tok_prob_shape", -3), ("tok_prob_dtype", -2), ("out_overlaps_tok_prob", -6),
                                         ("null_tok_prob", -1)])
def test_update_ranked_rejects(case, status):
    from paper_2608_02625_gb300.binding import lib
    d = dict(tok=T(I32, [2, 8], 1 * MB), msk=T(U8, [2, 8], 2 * MB), am=T(I32, [2, 8], 3 * MB),
             cf=T(F32, [2, 8], 4 * MB), tp=T(F32, [2, 8], 10 * MB), nt=T(I32, [2, 8], 5 * MB),
             nm=T(U8, [2, 8], 6 * MB), ne=T(I32, [2], 7 * MB))
    if case == "tok_prob_shape":
        d["tp"] = T(F32, [2, 9], 10 * MB)
    elif case == "tok_prob_dtype":
        d["tp"] = T(I32, [2, 8], 10 * MB)
    elif case == "out_overlaps_tok_prob":
        d["nt"] = T(I32, [2, 8], 10 * MB)
    elif case == "null_tok_prob":
        d["tp"] = None
    r = lambda x: ctypes.byref(x) if x is not None else None
    assert lib.dlm_refine_update_ranked(r(d["tok"]), r(d["msk"]), r(d["am"]), r(d["cf"]), r(d["tp"]), r(P()),
                                        r(d["nt"]), r(d["nm"]), r(d["ne"])) == status


def test_masked_attention_rejects():
    from paper_2608_02625_gb300.binding import lib
    q, k, v, sl, o = good_attn()
    pl = T(I32, [2], 6 * MB)
    r = ctypes.byref
    assert lib.dlm_attn_masked(r(q), r(k), r(v), r(sl), r(pl), 3, 64, r(o)) == -6         # unknown mode
    assert lib.dlm_attn_masked(r(q), r(k), r(v), r(sl), r(pl), 1, 0, r(o)) == -6          # block < 1
    assert lib.dlm_attn_masked(r(q), r(k), r(v), r(sl), r(T(I32, [3], 6 * MB)), 1, 64, r(o)) == -3
    assert lib.dlm_attn_masked(r(q), r(k), r(v), r(sl), r(T(F32, [2], 6 * MB)), 2, 64, r(o)) == -2


def test_selftest_rejects_budget_outside_range():
    so = ctypes.CDLL(os.path.join(PKG, "libdlmrefine.so"))
    so.dlm_selftest_wait_timeout.argtypes = [ctypes.c_int64]
    for budget in (0, 999, 1000000001, -5):
        assert so.dlm_selftest_wait_timeout(budget) == -6   # DLM_ERR_ARG, nothing launched


def test_checked_build_exports_its_test_hooks(tmp_path):
    """A DLM_CHECK_BOUNDS build exports what dlmrefine.h and dlmrefine_checked.h
    declare; the default build has none of the checked-only hooks."""
    from paper_2608_02625_gb300 import build
    build.build(check_bounds=True, out_dir=str(tmp_path))
    checked = ctypes.CDLL(str(tmp_path / "libdlmrefine.so"))
    default = ctypes.CDLL(os.path.join(PKG, "libdlmrefine.so"))
    hooks = declared_functions("dlmrefine_checked.h")
    assert hooks == ["dlm_checked_fill_static_scratch", "dlm_checked_set_wait_budget"]
    for n in declared_functions("dlmrefine.h") + hooks:
        assert hasattr(checked, n), f"checked build does not export {n}"
    for n in hooks:
        assert not hasattr(default, n), f"default build exports the test hook {n}"
    checked.dlm_checked_fill_static_scratch.argtypes = [ctypes.c_int32]
    assert checked.dlm_checked_fill_static_scratch(256) == -6
    checked.dlm_checked_set_wait_budget.argtypes = [ctypes.c_int64]
    assert checked.dlm_checked_set_wait_budget(99) == -6 and checked.dlm_checked_set_wait_budget(2000000001) == -6
    assert checked.dlm_checked_set_wait_budget(2000000000) == 0


def test_attn_tiles_per_unit_setting():
    from paper_2608_02625_gb300.binding import lib
    for bad in (-1, 3, 1 << 20):
        assert lib.dlm_set_attn_tiles_per_unit(bad) == -6
        assert b"dlm_set_attn_tiles_per_unit" in lib.dlm_last_error()
    for ok in (1, 2, 0):
        assert lib.dlm_set_attn_tiles_per_unit(ok) == 0
