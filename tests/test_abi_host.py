"""CPU checks of the C ABI: the library builds, loads and exports every symbol that
include/lilicorr.h declares, and its host-side logic (parameter count, argument and
shape validation, workspace sizing) behaves, without touching a GPU."""
import ctypes
import os
import re

import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = [os.path.join(ROOT, "include", h) for h in ("lilicorr.h", "lilicorr_testing.h")]


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_20530_gb300 as ll
    return ll.lib()


def declared_functions():
    src = "".join(open(h).read() for h in HEADERS)
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(lilicorr_[a-z_0-9]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for want in ("lilicorr_topk_lse", "lilicorr_embed_in_out", "lilicorr_pair_scores",
                 "lilicorr_greedy_walk", "lilicorr_select_block", "lilicorr_head_create",
                 "lilicorr_head_destroy", "lilicorr_workspace_bytes"):
        assert want in names


def test_every_declared_symbol_is_exported(lib):
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def _desc(**kw):
    import paper_2608_20530_gb300 as ll
    base = dict(H=4096, D=1024, d=1024, n_heads=8, ffn=2048, n_layers=2, L=15, K=8, V=151936,
                n_tgt=5, dtype=ll.BF16)
    base.update(kw)
    return ll.HeadDesc(**base)


def test_param_count_agrees_with_oracle_and_paper(lib):
    for H in (4096, 2560):
        n = lib.lilicorr_head_param_count(ctypes.byref(_desc(H=H)))
        assert n == oracle.param_count(H, 1024, 1024, 2048, 8, 15, 8)
    assert round(lib.lilicorr_head_param_count(ctypes.byref(_desc())) / 1e6, 2) == 36.76
    assert round(lib.lilicorr_head_param_count(ctypes.byref(_desc(H=2560))) / 1e6, 2) == 32.04


def test_invalid_descs_are_rejected(lib):
    for bad in (dict(K=0), dict(K=33), dict(L=0), dict(D=1004), dict(n_heads=7), dict(H=4095), dict(dtype=7),
                dict(K=8, V=4), dict(L=64, K=16)):
        assert lib.lilicorr_head_param_count(ctypes.byref(_desc(**bad))) == 0
    h = ctypes.c_void_p()
    blob = (ctypes.c_float * 4)()
    st = lib.lilicorr_head_create(ctypes.byref(_desc(K=0)), blob, blob, ctypes.byref(h))
    assert st == 2 and not h.value
    st = lib.lilicorr_head_create(ctypes.byref(_desc(dtype=9)), blob, blob, ctypes.byref(h))
    assert st == 3


def test_topk_argument_checks_need_no_gpu(lib):
    f = lib.lilicorr_topk_lse
    assert f(None, 0, 4, 10, 11, None, None, None, None, 0, None) == 2   # K > V
    assert f(None, 0, 4, 10, 0, None, None, None, None, 0, None) == 2    # K = 0
    assert f(None, 0, 4, 100, 33, None, None, None, None, 0, None) == 2  # K > MAX_K
    assert f(None, 5, 4, 10, 3, None, None, None, None, 0, None) == 3    # dtype
    assert f(None, 0, 0, 10, 3, None, None, None, None, 0, None) == 0    # no rows: nothing to do
    assert f(None, 0, 4, 10, 3, None, None, None, None, 0, None) == 1    # null pointers
    assert lib.lilicorr_topk_lse_workspace_bytes(4, 10, 11) == 0


def test_pair_and_walk_argument_checks(lib):
    assert lib.lilicorr_pair_scores(1, 0, 4, 8, None, None, None, None, None, None) == 2
    assert lib.lilicorr_pair_scores(1, 4, 33, 8, None, None, None, None, None, None) == 2
    assert lib.lilicorr_pair_scores(0, 4, 4, 8, None, None, None, None, None, None) == 0
    assert lib.lilicorr_pair_scores(1, 4, 4, 8, None, None, None, None, None, None) == 1
    assert lib.lilicorr_greedy_walk(1, 4, 0, None, None, None, None, None, None, None) == 2
    assert lib.lilicorr_greedy_walk(1, 4, 4, None, None, None, None, None, None, None) == 1


def test_status_strings(lib):
    for s in range(8):
        assert lib.lilicorr_status_str(s)
    assert lib.lilicorr_version() >= 1


def test_widened_calls_check_arguments_before_launching(lib):
    """Shape and argument errors come back synchronously, before any launch: the exact
    path, the local softmax, the path diagnostics, coverage/acceptance, the vocabulary
    shards and the fused LM head."""
    bp = lib.lilicorr_best_path
    assert bp(1, 0, 4, None, None, None, 8.0, None, None, None, None) == 2          # L = 0
    assert bp(1, 65, 4, None, None, None, 8.0, None, None, None, None) == 2         # L > MAX_L
    assert bp(1, 4, 33, None, None, None, 8.0, None, None, None, None) == 2         # K > MAX_K
    assert bp(1, 4, 4, None, None, None, 0.0, None, None, None, None) == 1          # sigma = 0
    assert bp(1, 4, 4, None, None, None, float("nan"), None, None, None, None) == 1
    assert bp(0, 4, 4, None, None, None, 8.0, None, None, None, None) == 0          # no work
    assert bp(1, 4, 4, None, None, None, 8.0, None, None, None, None) == 1          # nulls

    ls = lib.lilicorr_local_softmax
    assert ls(-1, 4, 4, None, None, 8.0, None, None, None) == 2
    assert ls(1, 4, 4, None, None, -1.0, None, None, None) == 1
    assert ls(1, 4, 4, None, None, float("inf"), None, None, None) == 1
    assert ls(0, 4, 4, None, None, 8.0, None, None, None) == 0
    assert ls(1, 4, 4, None, None, 8.0, None, None, None) == 1

    pp = lib.lilicorr_path_probs
    assert pp(1, 4, 0, None, None, None, 8.0, None, None, None, None) == 2
    assert pp(1, 4, 4, None, None, None, 0.0, None, None, None, None) == 1
    assert pp(1, 4, 4, None, None, None, 8.0, None, None, None, None) == 1

    ba = lib.lilicorr_block_acceptance
    assert ba(1, 0, 4, None, None, None, None, None, None, None) == 2
    assert ba(0, 4, 4, None, None, None, None, None, None, None) == 0
    assert ba(1, 4, 4, None, None, None, None, None, None, None) == 1

    part, merge = lib.lilicorr_topk_lse_partial, lib.lilicorr_topk_lse_merge
    assert part(None, 5, 4, 100, 8, 0, None, None, 0, None) == 3                   # dtype
    assert part(None, 0, 4, 100, 0, 0, None, None, 0, None) == 2                   # K = 0
    assert part(None, 0, 4, 100, 8, -1, None, None, 0, None) == 1                  # id offset
    assert part(None, 0, 4, 100, 8, 2**31 - 50, None, None, 0, None) == 1          # ids overflow
    assert part(None, 0, 0, 100, 8, 0, None, None, 0, None) == 0
    assert part(None, 0, 4, 100, 8, 0, None, None, 0, None) == 1
    assert merge(None, 0, 4, 8, None, None, None, None, None) == 2                 # P = 0
    assert merge(None, 1025, 4, 8, None, None, None, None, None) == 2              # P*K > 8192
    assert merge(None, 2, 0, 8, None, None, None, None, None) == 0
    assert merge(None, 2, 4, 8, None, None, None, None, None) == 1
    assert lib.lilicorr_topk_partial_bytes(0) == 0 and lib.lilicorr_topk_partial_bytes(33) == 0
    assert lib.lilicorr_topk_partial_bytes(8) >= 8 + 8 * 8                         # m, s, keys

    lm = lib.lilicorr_lm_head_topk
    assert lm(None, None, 4, 4096, 4, 8, None, None, None, None, 0, None) == 2     # K > V
    assert lm(None, None, 4, 4096, 100, 0, None, None, None, None, 0, None) == 2   # K = 0
    assert lm(None, None, 0, 4096, 100, 8, None, None, None, None, 0, None) == 0
