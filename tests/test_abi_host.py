"""The C-ABI library builds, loads and validates arguments on the host (no GPU)."""
import ctypes
import os
import re

import pytest

import paper_2609_32046_gb300 as cb
from paper_2609_32046_gb300 import binding
from paper_2609_32046_gb300.build import build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "cacheback.h")


@pytest.fixture(scope="module")
def lib():
    build()
    return binding.load_library()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(cb_[a-z_]+)\s*\(", src)))


def test_header_and_binding_agree():
    assert declared_functions() == sorted(binding.EXPORTED)


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_budget_matches_the_paper_rule(lib):
    # App. C.2: B_i = ceil(T_i / r), keep = 1/r, in double
    assert cb.budget(8192, 0.25) == 2048
    assert cb.budget(8192, 0.10) == 820
    assert cb.budget(65536, 0.10) == 6554
    assert cb.budget(16384, 0.25) == 4096
    assert cb.budget(100, 0.0) == 0
    assert cb.budget(100, 1.5) == 100
    assert cb.budget(0, 0.5) == 0


def _cfg(lib, **kw):
    c = binding.cb_config()
    lib.cb_config_init(ctypes.byref(c))
    base = dict(n_layers=2, n_q_heads=4, n_kv_heads=2, head_dim=64, max_query_tokens=16, max_positions=512,
                max_senders=1)
    base.update(kw)
    for k, v in base.items():
        setattr(c, k, v)
    return c


def test_chain_budget_matches_the_paper_rule(lib):
    """App. C.2's two chain budgets, library against the oracle's restatement."""
    import oracle
    for T_old in (0, 1, 41, 2048, 6554):
        for T_new in (0, 1, 40, 777, 25000, 61000):
            for keep in (0.1, 0.25, 1 / 3, 0.5):
                assert cb.chain_budget(T_old, T_new, keep) == oracle.chain_budget(T_old, T_new, keep)
            for B_max in (0, 41, 4096, 10 ** 7):
                assert cb.chain_budget(T_old, T_new, mode="fixed", B_max=B_max) == \
                    oracle.chain_budget(T_old, T_new, mode="fixed", B_max=B_max)
    assert cb.chain_budget(2048, 25000, 0.25) == 2048 + 6250          # inherited rows all count
    assert lib.cb_chain_budget(-1, 5, 0.5, 0, 0) == -1 and lib.cb_chain_budget(5, 5, 0.5, 2, 0) == -1
    assert lib.cb_chain_budget(5, 5, 0.5, 1, -1) == -1


def test_defaults_follow_the_paper(lib):
    c = binding.cb_config()
    lib.cb_config_init(ctypes.byref(c))
    assert (c.p, c.alpha, c.pool_width, c.span_width, c.n_sink, c.n_latent) == (2.0, 2.0, 7, 16, 1, 40)


@pytest.mark.parametrize("kw,status", [
    (dict(n_q_heads=6, n_kv_heads=4), binding.CB_ESHAPE),      # Hq % Hkv != 0
    (dict(n_q_heads=16, n_kv_heads=2), binding.CB_ESHAPE),     # G = 8 unsupported
    (dict(head_dim=96), binding.CB_ESHAPE),
    (dict(n_layers=0), binding.CB_ESHAPE),
    (dict(max_query_tokens=0), binding.CB_ESHAPE),
    (dict(max_query_tokens=5000), binding.CB_ESHAPE),
    (dict(max_positions=0), binding.CB_ESHAPE),
    (dict(max_senders=0), binding.CB_ESHAPE),
    (dict(p=1.0), binding.CB_EINVAL),
    (dict(p=float("nan")), binding.CB_EINVAL),
    (dict(alpha=-1.0), binding.CB_EINVAL),
    (dict(pool_width=6), binding.CB_EINVAL),
    (dict(pool_width=17), binding.CB_EINVAL),
    (dict(span_width=0), binding.CB_EINVAL),
    (dict(span_width=1000), binding.CB_EINVAL),
    (dict(n_latent=-1), binding.CB_EINVAL),
    (dict(softmax_scale=-1.0), binding.CB_EINVAL),
])
def test_create_rejects_bad_configs_before_touching_a_device(lib, kw, status):
    c = _cfg(lib, **kw)
    h = ctypes.c_void_p()
    assert lib.cb_create(ctypes.byref(c), ctypes.byref(h)) == status
    assert not h.value
    assert lib.cb_last_error(None)


def test_null_arguments(lib):
    h = ctypes.c_void_p()
    assert lib.cb_create(None, ctypes.byref(h)) == binding.CB_EINVAL
    assert lib.cb_create(ctypes.byref(_cfg(lib)), None) == binding.CB_EINVAL
    assert lib.cb_score(None, 1, None, None, None, None) == binding.CB_EINVAL
    assert lib.cb_select(None, 1, None, None, None, None, None) == binding.CB_EINVAL
    assert lib.cb_compact(None, 1, None, None, None, None, None, 0, None, 0, 0, None) == binding.CB_EINVAL
    lib.cb_destroy(None)
    assert lib.cb_scratch_bytes(None) == 0


def test_no_device_fails_loudly(lib):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    h = ctypes.c_void_p()
    assert lib.cb_create(ctypes.byref(_cfg(lib)), ctypes.byref(h)) == binding.CB_ECUDA
    with pytest.raises(cb.CBError):
        cb.CacheBack(2, 4, 2, 64, 16, 512)


def test_missing_library_raises(tmp_path):
    with pytest.raises(ImportError):
        binding.load_library(str(tmp_path / "libcacheback.so"))
