"""Host-side checks of the C ABI that need no GPU: the library loads, exports
every entry point include/wici.h declares, plans buffer sizes and rejects bad
configurations and arguments before touching a device."""
import ctypes
import os
import re

import pytest

import gen
from paper_2608_24204_gb300 import build, wici

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build()


def declared_entry_points():
    with open(os.path.join(ROOT, "include", "wici.h")) as f:
        src = f.read()
    return sorted(set(re.findall(r"^\s*(?:int|int32_t|void|const char \*)\s*(wici_\w+)\(", src, re.M)))


def test_library_exports_every_declared_entry_point():
    names = declared_entry_points()
    assert len(names) == 21
    L = wici.lib()
    for n in names:
        assert hasattr(L, n), n
    assert sorted(wici.EXPORTS) == names


def test_sizes_match_the_packed_layout():
    cfg = wici.make_config(gen.LLAMA_8B, max_tokens=8448, max_chunk=2048)
    s = wici.wici_get_sizes(cfg)
    params = sum(r * c for _, (r, c), _ in gen.tensor_specs(gen.LLAMA_8B))
    assert params * 2 <= s.weight_bytes <= params * 2 + 1_000_000
    assert s.kv_bytes == 32 * (8448 // 16) * 2 * 8 * 16 * 128 * 2
    assert s.workspace_bytes > 2048 * 14336 * 4
    tied = wici.wici_get_sizes(wici.make_config(gen.LLAMA_1B, 640))
    p1 = sum(r * c for _, (r, c), _ in gen.tensor_specs(gen.LLAMA_1B))
    assert p1 * 2 <= tied.weight_bytes <= p1 * 2 + 1_000_000   # the LM head aliases the embedding


def test_q8_sizes_hold_codes_and_block_scales():
    # the seven per-layer matrices at 17/16 bytes per parameter (codes + one fp16
    # scale per 32), everything else bf16; the prefill workspace adds one matrix
    # (the largest, gate|up) as three bf16 terms
    cfg = gen.LLAMA_8B
    b = wici.wici_get_sizes(wici.make_config(cfg, max_tokens=1296, max_chunk=1024))
    q = wici.wici_get_sizes(wici.make_config(cfg, max_tokens=1296, max_chunk=1024, q8=True))
    per_layer = sum(r * c for n, (r, c), _ in gen.tensor_specs(cfg)
                    if n.startswith("layers.0.") and n.split(".")[-1] in ("wq", "wk", "wv", "wo", "wg", "wu", "wd"))
    saved = cfg.n_layers * per_layer * (2 - 17 / 16)
    assert abs((b.weight_bytes - q.weight_bytes) - saved) < 1_000_000
    assert q.workspace_bytes - b.workspace_bytes >= 3 * 2 * (2 * cfg.ffn_dim * cfg.hidden)
    assert q.kv_bytes == b.kv_bytes


def test_conv_shape_checks_and_workspace_size():
    s = wici.wici_conv_shape(4, 1024, 224, 224, 1024)
    assert wici.wici_conv_workspace_bytes(s) == 256 + 9 * 1024 * 1024 * 2
    for bad in ((4, 1000, 224, 224, 1024), (4, 1024, 223, 224, 1024), (0, 256, 8, 8, 256)):
        with pytest.raises(wici.WiciError) as e:
            wici.wici_conv_workspace_bytes(wici.wici_conv_shape(*bad))
        assert e.value.status == wici.WICI_E_ARG


def test_q8_rejects_widths_that_are_not_multiples_of_256():
    with pytest.raises(wici.WiciError) as e:
        wici.wici_get_sizes(wici.make_config(gen.TINY, 64, q8=True))      # ffn 688
    assert e.value.status == wici.WICI_E_ARG and "256" in str(e.value)
    wici.wici_get_sizes(wici.make_config(gen.TINY.with_(ffn_dim=768), 64, q8=True))


@pytest.mark.parametrize("field,value", [("head_dim", 96), ("n_kv_heads", 3), ("page_tokens", 32),
                                         ("hidden", 260), ("max_chunk", 0), ("n_layers", 0),
                                         ("rms_eps", 0.0), ("qkv_bias", 2)])
def test_bad_config_is_rejected(field, value):
    cfg = wici.make_config(gen.TINY, 64)
    setattr(cfg, field, value)
    with pytest.raises(wici.WiciError) as e:
        wici.wici_get_sizes(cfg)
    assert e.value.status == wici.WICI_E_ARG
    assert "config" in str(e.value)


def test_null_arguments_are_rejected_without_a_device():
    L = wici.lib()
    cfg = wici.make_config(gen.TINY, 64)
    assert L.wici_get_sizes(None, None) == wici.WICI_E_ARG
    out = ctypes.c_void_p()
    assert L.wici_create(ctypes.byref(cfg), None, None, None, None, ctypes.byref(out)) == wici.WICI_E_ARG
    assert L.wici_create(ctypes.byref(cfg), None, 256, 512, 7, ctypes.byref(out)) == wici.WICI_E_ARG  # unaligned
    assert "aligned" in wici.wici_last_error(None)
    assert L.wici_prefill(None, None, 0, None, None) == wici.WICI_E_ARG
    assert L.wici_decode_step(None, 0, None, None) == wici.WICI_E_ARG
    assert L.wici_kv_len(None) == wici.WICI_E_ARG
    L.wici_destroy(None)


def test_flops_and_bytes_accounting_of_the_headline_workload():
    assert gen.prefill_flops(gen.LLAMA_8B, 1024) == pytest.approx(14.57e12, rel=1e-3)
    total = sum(gen.prefill_flops(gen.LLAMA_8B, 2048, P) for P in (0, 2112, 4224, 6336))
    assert total == pytest.approx(132.36e12, rel=1e-3)
    avg = sum(gen.decode_bytes_per_token(gen.LLAMA_8B, 1024 + i) for i in range(1, 257)) / 256
    assert avg == pytest.approx(15.161e9, rel=1e-3)
