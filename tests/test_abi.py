"""The C ABI library: builds, exports every entry point of include/pced.h, and
rejects invalid host arguments before touching the device.  No GPU needed:
every call here fails host-side validation."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
FAKE = 1 << 12  # non-null, aligned; never dereferenced because validation fails first


@pytest.fixture(scope="module")
def L():
    from paper_2601_08670_gb300 import build
    build.build()
    import paper_2601_08670_gb300 as pced
    return pced.lib()


def declared_functions():
    src = open(os.path.join(ROOT, "include", "pced.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(pced_[a-z_]+)\s*\(", src)))


def test_every_declared_symbol_is_exported(L):
    names = declared_functions()
    assert len(names) >= 11
    for n in names:
        assert hasattr(L, n), n


def test_status_strings(L):
    assert L.pced_status_string(0) == b"ok"
    assert L.pced_status_string(3) == b"unsupported shape"


def test_attention_rejects_bad_arguments(L):
    f = L.pced_decode_attention
    # null q
    assert f(None, FAKE, FAKE, 1 << 20, FAKE, FAKE, FAKE, 2, 8, 2, 64, 100, 0.1, FAKE, FAKE, 1 << 30, None) == 1
    # Hq not a multiple of Hkv
    assert f(FAKE, FAKE, FAKE, 1 << 20, FAKE, FAKE, FAKE, 2, 7, 2, 64, 100, 0.1, FAKE, FAKE, 1 << 30, None) == 1
    # unsupported head dim
    assert f(FAKE, FAKE, FAKE, 96 << 10, FAKE, FAKE, FAKE, 2, 8, 2, 96, 100, 0.1, FAKE, FAKE, 1 << 30, None) == 3
    # group of 16 query heads per kv head
    assert f(FAKE, FAKE, FAKE, 1 << 20, FAKE, FAKE, FAKE, 2, 32, 2, 64, 100, 0.1, FAKE, FAKE, 1 << 30, None) == 3
    # misaligned cache
    assert f(FAKE, FAKE + 2, FAKE, 1 << 20, FAKE, FAKE, FAKE, 2, 8, 2, 64, 100, 0.1, FAKE, FAKE, 1 << 30, None) == 1
    # workspace too small
    assert f(FAKE, FAKE, FAKE, 1 << 20, FAKE, FAKE, FAKE, 2, 8, 2, 64, 100, 0.1, FAKE, FAKE, 16, None) == 2
    assert b"workspace" in L.pced_last_error()


def test_lm_head_rejects_bad_arguments(L):
    f = L.pced_lm_head_logprobs
    assert f(FAKE, FAKE, 4, 100, 1000, FAKE, FAKE, FAKE, 1 << 30, None) == 3  # d % 64 != 0
    assert f(FAKE, FAKE, 600, 128, 1000, FAKE, FAKE, FAKE, 1 << 30, None) == 3  # S > 512
    assert f(FAKE, FAKE, 0, 128, 1000, FAKE, FAKE, FAKE, 1 << 30, None) == 1
    assert f(FAKE, FAKE, 4, 128, 1000, FAKE, FAKE, FAKE, 8, None) == 2


def test_select_rejects_bad_arguments(L):
    f = L.pced_contrastive_select
    assert f(FAKE, FAKE, FAKE, 2.5, 0, 4, 100, FAKE, FAKE, FAKE, FAKE, 1 << 30, None) == 1
    assert f(FAKE, FAKE, FAKE, 2.5, 1, 300, 100, FAKE, FAKE, FAKE, FAKE, 1 << 30, None) == 3
    assert f(FAKE, FAKE, FAKE, float("nan"), 1, 4, 100, FAKE, FAKE, FAKE, FAKE, 1 << 30, None) == 1
    assert f(FAKE, FAKE, FAKE, 2.5, 1, 4, 100, FAKE, FAKE, FAKE, FAKE, 8, None) == 2


def test_adacad_beta_rejects_bad_arguments(L):
    f = L.pced_adacad_beta
    big = 1 << 30
    assert f(None, 1, 2, 100, FAKE, FAKE, big, None) == 1
    assert f(FAKE, 1, 2, 100, None, FAKE, big, None) == 1
    assert f(FAKE, 0, 2, 100, FAKE, FAKE, big, None) == 1
    assert f(FAKE, 1, 0, 100, FAKE, FAKE, big, None) == 1
    assert f(FAKE, 1, 2, 0, FAKE, FAKE, big, None) == 1
    assert f(FAKE + 2, 1, 2, 100, FAKE, FAKE, big, None) == 1  # misaligned
    assert f(FAKE, 1, 2, 100, FAKE, FAKE, 8, None) == 2        # workspace too small
    assert L.pced_adacad_beta_workspace_size(1, 2, 100) > 0


def test_relevance_rejects_bad_arguments(L):
    f = L.pced_relevance
    assert f(FAKE, 0, None, -1, 1e-8, FAKE, None) == 1      # n < 0
    assert f(FAKE, 2, None, 4, 1e-8, FAKE, None) == 1       # no such retrieval mode
    assert f(FAKE, 0, None, 4, -1.0, FAKE, None) == 1       # eps < 0
    assert f(FAKE, 0, None, 4, float("nan"), FAKE, None) == 1
    assert f(None, 0, None, 4, 1e-8, FAKE, None) == 1       # null scores
    assert f(FAKE, 1, FAKE + 2, 4, 1e-8, FAKE, None) == 1   # misaligned reranker logits
    assert f(None, 0, None, 0, 1e-8, None, None) == 0       # nothing to do


def test_step_rejects_bad_rope_and_block_arguments(L):
    import paper_2601_08670_gb300 as pced
    f = lambda a: L.pced_step(ctypes.byref(a), None)
    assert f(step_args(pced, rope_theta=-1.0)) == 1
    assert f(step_args(pced, rope_theta=float("inf"))) == 1
    assert f(step_args(pced, block_table=FAKE, block_rows=96, max_blocks=4)) == 1   # not a multiple of 64
    assert f(step_args(pced, block_table=FAKE, block_rows=64, max_blocks=0)) == 1
    assert f(step_args(pced, score_mode=2)) == 1
    assert f(step_args(pced, aggregation=3)) == 1
    assert f(step_args(pced, aggregation=-1)) == 1


def test_step_dynamic_beta_needs_its_output(L):
    import paper_2601_08670_gb300 as pced
    a = step_args(pced, beta_from_step=1)
    assert L.pced_step(ctypes.byref(a), None) == 1


def step_args(pced, **kw):
    dm = pced.dims(1, 8, 32, 32, 8, 128, 128256)
    a = pced.StepArgs()
    a.dims = dm
    for name in ("embed", "w_unembed", "k_cache", "v_cache", "kv_offset", "cap", "seq_len", "step", "history",
                 "beta", "r", "workspace"):
        setattr(a, name, FAKE)
    a.layer_elems = 1 << 24
    a.total_cap = 20000
    a.max_steps = 64
    a.gamma = 2.5
    a.attn_scale = 0.088
    a.rms_eps = 1e-6
    a.workspace_bytes = 1 << 40
    for k, v in kw.items():
        if k in ("B", "N", "L", "Hq", "Hkv", "D", "V"):
            setattr(a.dims, k, v)
        else:
            setattr(a, k, v)
    return a


def test_step_rejects_bad_arguments(L):
    import paper_2601_08670_gb300 as pced
    f = lambda a: L.pced_step(ctypes.byref(a), None)
    assert L.pced_step(None, None) == 1
    assert f(step_args(pced, embed=None)) == 1
    assert f(step_args(pced, Hkv=3)) == 1          # 32 % 3 != 0
    assert f(step_args(pced, Hq=8, Hkv=8)) == 1    # 2 * Hkv > Hq: no room for the appended V heads
    assert f(step_args(pced, D=96)) == 3
    assert f(step_args(pced, bos_token=128256)) == 1
    assert f(step_args(pced, workspace_bytes=100)) == 2
    # beyond the maxima: S = B (N + 1) > 512, N + 1 > 256 sequences per query
    assert f(step_args(pced, B=3, N=170)) == 3
    assert f(step_args(pced, B=1, N=256)) == 3


def test_step_host_io_rejects_bad_arguments(L):
    import paper_2601_08670_gb300 as pced
    f = lambda a, tok=None, exp=None, sc=None: L.pced_step_host_io(ctypes.byref(a), None, None, tok, exp, sc, None)
    assert L.pced_step_host_io(None, None, None, None, None, None, None) == 1
    # a host output needs its device output
    assert f(step_args(pced), tok=FAKE) == 1
    assert f(step_args(pced), exp=FAKE) == 1
    assert f(step_args(pced), sc=FAKE) == 1
    # not for an expert-partitioned call
    assert f(step_args(pced, key_out=FAKE, token_out=FAKE), tok=FAKE) == 1
    # the step's own validation applies
    assert f(step_args(pced, embed=None, token_out=FAKE), tok=FAKE) == 1
    assert f(step_args(pced, D=96)) == 3


def test_launch_count_and_kinds_follow_the_mode(L):
    import paper_2601_08670_gb300 as pced
    assert pced.step_launch_kinds(step_args(pced)) == ["attention", "lm_head", "select"]
    assert pced.step_launch_kinds(step_args(pced, beta_from_step=1)) == [
        "attention", "lm_head", "lse_finalize", "adacad_beta", "agg_select"]
    for rule in (pced.AGG_MOE, pced.AGG_POE):
        # the aggregation kernels read the raw logits: no finalise launch
        assert pced.step_launch_kinds(step_args(pced, aggregation=rule)) == [
            "attention", "lm_head", "agg_partials", "agg_select"]
        assert pced.step_launch_kinds(step_args(pced, aggregation=rule, beta_from_step=1)) == [
            "attention", "lm_head", "lse_finalize", "adacad_beta", "agg_partials", "agg_select"]
    a = step_args(pced, aggregation=pced.AGG_MOE)
    assert pced.step_launch_count(a) == 4
    assert L.pced_step_launch_kind(ctypes.byref(a), 4) is None
    assert L.pced_step_launch_kind(ctypes.byref(a), -1) is None
    assert L.pced_step_launch_count(None) == 0


def test_workspace_sizes(L):
    import paper_2601_08670_gb300 as pced
    dm = pced.dims(1, 8, 32, 32, 8, 128, 128256)
    assert pced.step_workspace_size(dm) > 0
    assert pced.step_workspace_size(pced.dims(1, 8, 32, 30, 8, 128, 100)) == 0
    assert L.pced_decode_attention_workspace_size(9, 32, 8, 128) > 0
    assert L.pced_lm_head_workspace_size(9, 128256) > 0


@pytest.mark.skipif(__import__("torch").cuda.is_available(), reason="only meaningful without a GPU")
def test_valid_call_without_device_reports_no_device(L):
    import torch  # noqa: F401
    assert L.pced_contrastive_select(FAKE, FAKE, FAKE, 2.5, 1, 4, 100, FAKE, FAKE, FAKE, FAKE, 1 << 30, None) == 5


def test_binding_rejects_bad_tensors_before_any_call(L):
    # the binding's own checks raise ValueError (also under python -O),
    # before the library or a device is touched
    import torch
    import paper_2601_08670_gb300 as pced
    with pytest.raises(ValueError):
        pced.relevance(torch.zeros(4, dtype=torch.float64))
    with pytest.raises(ValueError):
        pced.relevance(torch.zeros(4), rer_logits=torch.zeros(5))
    with pytest.raises(ValueError):
        pced.relevance(torch.zeros(4, 2).t())  # not contiguous
