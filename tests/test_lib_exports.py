"""Host-side checks of the C-ABI library: it builds, loads, exports every declared symbol and
validates arguments before touching a GPU (no compute calls here)."""
import ctypes as C
import os
import shutil

import pytest

from paper_2607_12422_gb300 import pbd, synth


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(pbd.LIB_PATH):
        if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
            pytest.skip("nvcc unavailable and libpbd.so not built")
        from paper_2607_12422_gb300 import build
        build.build()
    return pbd.load()


def test_every_declared_function_is_exported(lib):
    names = pbd.header_functions()
    assert "pbd_create" in names and "pbd_op_linear" in names and len(names) >= 18
    for n in names:
        assert hasattr(lib, n), n


def test_workspace_size_and_config_validation(lib):
    ok = pbd.make_config(synth.QWEN3_0_6B, 16, 1, 1024)
    n = lib.pbd_workspace_bytes(C.byref(ok))
    # at least the re-tiled weights (tied embedding once) and the KV cache
    assert n > 1_190_000_000
    bad = pbd.make_config(synth.QWEN3_0_6B, 16, 1, 1024)
    bad.head_dim = 96
    assert lib.pbd_workspace_bytes(C.byref(bad)) == 0
    bad = pbd.make_config(synth.QWEN3_0_6B, 16, 1, 1024)
    bad.page_size = 32
    assert lib.pbd_workspace_bytes(C.byref(bad)) == 0
    bad = pbd.make_config(synth.QWEN3_0_6B, 16, 1, 1024)
    bad.lora_rank = 64
    assert lib.pbd_workspace_bytes(C.byref(bad)) == 0
    tiny = pbd.make_config(synth.TINY, 16, 4, 256)
    assert 0 < lib.pbd_workspace_bytes(C.byref(tiny)) < 200_000_000
    # draft variants: early exit within the depth, at most 8 denoising steps, a 0/1 readout flag
    var = pbd.make_config(synth.TINY, 16, 4, 256, draft_layers=1, denoise_steps=2, anchored=False)
    assert lib.pbd_workspace_bytes(C.byref(var)) == lib.pbd_workspace_bytes(C.byref(tiny))
    # a CTA limit does not change the workspace (sized for 256 CTAs)
    capped = pbd.make_config(synth.TINY, 16, 4, 256, max_ctas=8)
    assert lib.pbd_workspace_bytes(C.byref(capped)) == lib.pbd_workspace_bytes(C.byref(tiny))
    for field, value in (("draft_layers", synth.TINY.n_layers + 1), ("draft_layers", -1), ("denoise_steps", 9),
                         ("draft_unanchored", 2), ("max_ctas", -1), ("max_ctas", 257)):
        bad = pbd.make_config(synth.TINY, 16, 4, 256)
        setattr(bad, field, value)
        assert lib.pbd_workspace_bytes(C.byref(bad)) == 0, field


def test_create_rejects_bad_arguments_without_gpu(lib):
    cfg = pbd.make_config(synth.TINY, 16, 1, 128)
    bw, aw = pbd.pbd_base_weights(), pbd.pbd_adapter_weights()
    out = C.c_void_p()
    assert lib.pbd_create(C.byref(cfg), C.byref(bw), C.byref(aw), None, 0, None, C.byref(out)) == 2
    assert b"workspace" in lib.pbd_last_error(None)
    assert lib.pbd_create(C.byref(cfg), C.byref(bw), C.byref(aw), 0x1001, 1 << 30, None, C.byref(out)) == 2
    cfg.block_D = 0
    assert lib.pbd_create(C.byref(cfg), C.byref(bw), C.byref(aw), 0x100000, 1 << 30, None, C.byref(out)) == 1
    assert b"block_D" in lib.pbd_last_error(None)
    assert not out.value
    # op entry points size-check before any launch
    assert lib.pbd_op_linear_workspace_bytes(17, 1000, 128, 16) == 0
    assert lib.pbd_op_linear_workspace_bytes(17, 1024, 100, 16) == 0
    assert lib.pbd_op_linear_workspace_bytes(17, 1024, 128, 16) > 0
    assert lib.pbd_op_lm_head_workspace_bytes(300, 1024, 4096) == 0
    assert lib.pbd_version().startswith(b"pbd sm_103a")


def test_op_status_validates_arguments_without_gpu(lib):
    code = C.c_int32(-1)
    assert lib.pbd_op_status(None, None, C.byref(code)) == 1 and code.value == 0
    assert lib.pbd_op_status(0x100010, None, None) == 1  # not 1024-byte aligned
    assert b"pbd_op_status" in lib.pbd_op_last_error()


def test_state_calls_need_a_context(lib):
    assert lib.pbd_draft_block(None, None, None) == 1
    assert lib.pbd_sync(None) == 1
