"""The C-ABI library builds, loads and exports every symbol include/kvblend.h declares;
host-only entry points and argument validation work without a GPU."""
import ctypes as C
import os
import re

import numpy as np
import pytest

from oracle import llama
from oracle.llama import Shape
from paper_2609_09768_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def kvb():
    from paper_2609_09768_gb300 import build, kvblend
    build.build()
    kvblend.lib()
    return kvblend


def header_functions():
    text = open(os.path.join(ROOT, "include", "kvblend.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(kvb_[a-z0-9_]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(kvb):
    names = header_functions()
    assert len(names) >= 15
    lib = C.CDLL(kvb.lib_path())
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(kvb.EXPORTED), set(names) ^ set(kvb.EXPORTED)


def test_status_strings_and_version(kvb):
    L = kvb.lib()
    assert L.kvb_version() >= 100
    for code, text in kvb.STATUS.items():
        assert L.kvb_status_string(code).decode() == text


def test_rope_table_matches_oracle(kvb):
    for shape in (synth.TINY, synth.LLAMA8B, synth.YARN_GQA7_TINY, synth.YARN_GQA7):
        cfg = kvb.config(shape)
        cos, sin = kvb.rope_table_fill(cfg, 130000)
        pos = np.array([0, 1, 2, 511, 8191, 8192, 65537, 124031, 129999])
        c, s = llama.rope_cos_sin(Shape.of(shape), pos)
        assert np.max(np.abs(cos[pos] - c)) < 1e-6 and np.max(np.abs(sin[pos] - s)) < 1e-6


def test_attention_scale_matches_oracle(kvb):
    """1/sqrt(D), times YaRN's (0.1 ln s + 1)^2 for the YaRN shapes."""
    for shape in (synth.TINY, synth.LLAMA8B, synth.YARN_GQA7_TINY, synth.YARN_GQA7):
        got = kvb.attention_scale(kvb.config(shape))
        assert abs(got - llama.logit_scale(Shape.of(shape))) <= 1e-7 * got
    assert kvb.attention_scale(kvb.config(synth.YARN_GQA7)) > 1.0 / np.sqrt(128) * 1.2


def test_config_validation_of_rope_scaling_and_groups(kvb):
    L = kvb.lib()
    n = C.c_size_t(0)
    cfg = kvb.config(synth.YARN_GQA7)           # seven q heads per kv head: accepted
    assert L.kvb_workspace_size(C.byref(cfg), 100, C.byref(n)) == kvb.KVB_OK
    assert L.kvb_decode_workspace_size(C.byref(cfg), 100, C.byref(n)) == kvb.KVB_OK
    bad = kvb.config(synth.YARN_GQA7)
    bad.rope_scaling = 3
    assert L.kvb_workspace_size(C.byref(bad), 100, C.byref(n)) == kvb.KVB_ERR_INVALID_ARG
    bad = kvb.config(synth.YARN_GQA7)
    bad.rs_factor = 0.5                         # YaRN extends the context: s >= 1
    assert L.kvb_workspace_size(C.byref(bad), 100, C.byref(n)) == kvb.KVB_ERR_INVALID_ARG
    bad = kvb.config(synth.YARN_GQA7)
    bad.rs_high = bad.rs_low
    assert L.kvb_workspace_size(C.byref(bad), 100, C.byref(n)) == kvb.KVB_ERR_INVALID_ARG
    three = kvb.config(synth.LLAMA8B)           # 3 q heads per kv head: prefill and decode
    three.n_q_heads, three.n_kv_heads = 24, 8
    assert L.kvb_workspace_size(C.byref(three), 100, C.byref(n)) == kvb.KVB_OK
    assert L.kvb_decode_workspace_size(C.byref(three), 100, C.byref(n)) == kvb.KVB_OK
    wide = kvb.config(synth.LLAMA8B)            # 16 q heads per kv head: prefill yes, decode not built
    wide.n_q_heads, wide.n_kv_heads = 32, 2
    assert L.kvb_workspace_size(C.byref(wide), 100, C.byref(n)) == kvb.KVB_OK
    assert L.kvb_decode_workspace_size(C.byref(wide), 100, C.byref(n)) == kvb.KVB_ERR_UNSUPPORTED


def test_workspace_size_grows_with_rows(kvb):
    cfg = kvb.config(synth.LLAMA8B)
    a, b = kvb.workspace_size(cfg, 1000), kvb.workspace_size(cfg, 124032)
    assert 0 < a < b
    # residuals (2 x fp32), bf16 activations and the MLP intermediate for 124k rows
    assert b > 124032 * 4096 * (4 + 4 + 2) + 124032 * 14336 * 2


def test_host_validation_rejects_bad_arguments(kvb):
    L = kvb.lib()
    cfg = kvb.config(synth.TINY)
    # NULL config / pointers are rejected before any device work
    assert L.kvb_rope_table_fill(None, 10, None, None) == kvb.KVB_ERR_INVALID_ARG
    assert L.kvb_selective_prefill(None, None, None, None, None, None, None, None, 0, 0, 0, 0.15, 1, None, 0, None,
                                   None, None, None, None, 0, None) == kvb.KVB_ERR_INVALID_ARG
    assert b"config is NULL" in L.kvb_last_error()
    bad = kvb.config(synth.TINY)
    bad.head_dim = 96
    n = C.c_size_t(0)
    assert L.kvb_workspace_size(C.byref(bad), 10, C.byref(n)) == kvb.KVB_ERR_UNSUPPORTED
    bad = kvb.config(synth.TINY)
    bad.n_kv_heads = 3
    assert L.kvb_workspace_size(C.byref(bad), 10, C.byref(n)) == kvb.KVB_ERR_UNSUPPORTED
    # k > n_ctx, misaligned leading dims
    assert L.kvb_hkvd_select(None, 128, None, 128, 10, 128, 11, None, None, None, 0, None) == kvb.KVB_ERR_INVALID_ARG
    assert L.kvb_hkvd_select(None, 12, None, 12, 10, 12, 1, None, None, None, 0, None) == kvb.KVB_ERR_INVALID_ARG
    # misaligned pointer
    assert L.kvb_kv_scatter(8, 16, 16, 1, 128, 16, 16, 4, None) == kvb.KVB_ERR_INVALID_ARG
    assert b"aligned" in L.kvb_last_error()
    # r outside [0, 1] and a check layer outside [1, L]
    mw = kvb.ModelStruct()
    assert L.kvb_selective_prefill(C.byref(cfg), C.byref(mw), None, None, None, None, None, None, 1, 10, 2, 1.5, 1,
                                   None, 0, None, None, None, None, None, 0, None) == kvb.KVB_ERR_INVALID_ARG
    assert L.kvb_debug_wait_timeout(None, 0, 10**6, None) == kvb.KVB_ERR_INVALID_ARG
    # empty inputs are valid no-ops
    assert L.kvb_kv_scatter(None, None, None, 0, 128, None, None, 4, None) == kvb.KVB_OK
    assert L.kvb_hkvd_select(None, 128, None, 128, 0, 128, 0, None, None, None, 0, None) == kvb.KVB_OK


def test_binding_fails_loudly_without_library(monkeypatch):
    from paper_2609_09768_gb300 import kvblend
    monkeypatch.setattr(kvblend, "_LIB", None)
    monkeypatch.setattr(kvblend, "LIB", "/nonexistent/libkvblend.so")
    with pytest.raises(RuntimeError, match="not built"):
        kvblend.lib()


def test_shape_from_published_config_layout():
    """The config reader maps the common checkpoint JSON layout onto ModelShape (values here
    are made up for the test)."""
    base = {"hidden_size": 1792, "num_attention_heads": 14, "num_key_value_heads": 2, "intermediate_size": 4864,
            "num_hidden_layers": 3, "vocab_size": 5000, "rms_norm_eps": 1e-6, "rope_theta": 1e6}
    s = synth.shape_from_config(dict(base, rope_scaling={"type": "yarn", "factor": 4.0,
                                                         "original_max_position_embeddings": 2048}, qkv_bias=True))
    assert (s.hidden, s.n_q_heads, s.n_kv_heads, s.head_dim, s.mlp_dim, s.n_layers, s.vocab) == \
        (1792, 14, 2, 128, 4864, 3, 5000)
    assert (s.rope_scaling, s.rs_factor, s.rs_low, s.rs_high, s.rs_orig_ctx, s.qkv_bias) == (2, 4.0, 1.0, 32.0, 2048, True)
    assert s == synth.YARN_GQA7.with_layers(3).__class__(**{**synth.YARN_GQA7.__dict__, "n_layers": 3, "vocab": 5000})
    l3 = synth.shape_from_config(dict(base, rope_scaling={"rope_type": "llama3", "factor": 8.0, "low_freq_factor": 1.0,
                                                          "high_freq_factor": 4.0,
                                                          "original_max_position_embeddings": 8192},
                                      attention_bias=False))
    assert (l3.rope_scaling, l3.rs_factor, l3.rs_low, l3.rs_high, l3.rs_orig_ctx, l3.qkv_bias) == (1, 8.0, 1.0, 4.0, 8192, False)
    plain = synth.shape_from_config(dict(base, head_dim=64))
    assert plain.rope_scaling == 0 and plain.head_dim == 64
    with pytest.raises(ValueError):
        synth.shape_from_config(dict(base, rope_scaling={"type": "dynamic", "factor": 2.0}))


def test_both_qkv_entry_points_validate_alike(kvb):
    """The workspace and the allocation-free QKV entry points accept and reject the same
    configurations (they share one validation); a failed call leaves a message, and the next
    successful validation step clears it."""
    L = kvb.lib()
    lw = kvb.LayerWeights(16, 16, 16, 16, 16, 16, 16, None)
    for hq, hkv in ((0, 2), (-2, 2), (4, 0)):
        bad = kvb.config(synth.TINY)
        bad.n_q_heads, bad.n_kv_heads = hq, hkv
        a = L.kvb_gather_rmsnorm_qkv(C.byref(bad), C.byref(lw), None, None, None, None, 4, None, None, None, None,
                                     8, None, 0, None)
        msg_a = L.kvb_last_error()
        b = L.kvb_gather_rmsnorm_qkv_noalloc(C.byref(bad), C.byref(lw), None, None, None, None, 4, None, None, None,
                                             None, 8, None, None)
        msg_b = L.kvb_last_error()
        assert a == b == kvb.KVB_ERR_INVALID_ARG, (hq, hkv, a, b)
        assert msg_a == msg_b and msg_a
    good = kvb.config(synth.TINY)
    # a bad eps / theta and an unknown scaling are rejected by both as well
    for field, value in (("rms_eps", -1.0), ("rope_theta", 0.0), ("rope_scaling", 9)):
        bad = kvb.config(synth.TINY)
        setattr(bad, field, value)
        a = L.kvb_gather_rmsnorm_qkv(C.byref(bad), C.byref(lw), None, None, None, None, 4, None, None, None, None,
                                     8, None, 0, None)
        b = L.kvb_gather_rmsnorm_qkv_noalloc(C.byref(bad), C.byref(lw), None, None, None, None, 4, None, None, None,
                                             None, 8, None, None)
        assert a == b == kvb.KVB_ERR_INVALID_ARG, field
    # with a valid config, m == 0 is a no-op for both and clears the previous message
    assert L.kvb_gather_rmsnorm_qkv(C.byref(good), C.byref(lw), None, None, None, None, 0, None, None, None, None, 0,
                                    None, 0, None) == kvb.KVB_OK
    assert L.kvb_last_error() == b""
    assert L.kvb_gather_rmsnorm_qkv_noalloc(C.byref(good), C.byref(lw), None, None, None, None, 0, None, None, None,
                                            None, 0, None, None) == kvb.KVB_OK
    assert L.kvb_last_error() == b""
    # a NULL rope table is rejected by both once there are rows to compute
    assert L.kvb_gather_rmsnorm_qkv(C.byref(good), C.byref(lw), None, 16, None, 16, 4, 16, 16, 16, None, 8, None, 0,
                                    None) == kvb.KVB_ERR_INVALID_ARG
    assert L.kvb_gather_rmsnorm_qkv_noalloc(C.byref(good), C.byref(lw), None, 16, None, 16, 4, 16, 16, 16, None, 8,
                                            None, None) == kvb.KVB_ERR_INVALID_ARG


def test_layer_taps_are_validated_before_any_launch(kvb):
    """A tap outside [0, n_layers] or one that needs more rows than its slots hold fails the
    call with INVALID_ARG before anything runs.  The device pointers here are stand-ins that
    validation only checks for alignment; no GPU is needed because nothing is launched."""
    L = kvb.lib()
    cfg = kvb.config(synth.TINY)                       # 2 layers
    fake = 1 << 20                                     # aligned, never dereferenced
    lws = (kvb.LayerWeights * cfg.n_layers)(*[kvb.LayerWeights(fake, fake, fake, fake, fake, fake, fake, None)
                                               for _ in range(cfg.n_layers)])
    mw = kvb.ModelStruct(C.cast(lws, C.POINTER(kvb.LayerWeights)), fake, fake)
    rope = kvb.RopeTableStruct(fake, fake, 1000)
    n = 300
    cache = kvb.KVCache(fake, fake, n, cfg.n_layers)

    def call(layer, rows_cap):
        layers = (C.c_int32 * 1)(layer)
        taps = kvb.LayerTapsStruct(1, layers, fake, rows_cap, None)
        return L.kvb_full_prefill(C.byref(cfg), C.byref(mw), C.byref(rope), C.byref(cache), None, fake, n, None,
                                  None, None, 0, None, C.byref(taps), None, 0, None)

    assert call(3, n) == kvb.KVB_ERR_INVALID_ARG and b"taps: layer 3 not in [0, 2]" in L.kvb_last_error()
    assert call(-1, n) == kvb.KVB_ERR_INVALID_ARG
    assert call(1, n - 1) == kvb.KVB_ERR_INVALID_ARG and b"carries 300 rows" in L.kvb_last_error()
    # a valid tap passes validation and the call stops at the (missing) workspace instead
    assert call(2, n) == kvb.KVB_ERR_WORKSPACE
