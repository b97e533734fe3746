"""pbd_op_linear_static: the block linear without a workspace, its scratch in the library's own
static device array.  Its output must match pbd_op_linear's on the same inputs, on calls made
back to back (the second call must see nothing of the first's scratch), and it must reject a
problem larger than the scratch before launching anything.  Named so that it runs after the
other test files; it also passes on its own."""
import ctypes as C
import os
import shutil

import numpy as np
import pytest

from paper_2607_12422_gb300 import pbd, synth

SCRATCH_BYTES = 16 << 20


def _need(M, K, N, r):
    """Scratch bytes of one call, from the size rule the header states."""
    s = K // 256 if K % 256 == 0 else 1
    return 2048 + (N // 128 + (1 if r > 0 else 0)) * (K // 64) * 16384 + 4 * s * M * (N + r)


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(pbd.LIB_PATH):
        if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
            pytest.skip("nvcc unavailable and libpbd.so not built")
        from paper_2607_12422_gb300 import build
        build.build()
    return pbd.load()


def test_oversize_and_bad_sizes_rejected_before_any_launch(lib):
    # 6144 x 1024 weight with r = 16: fits up to M = 39, not at M = 40
    assert _need(39, 1024, 6144, 16) <= SCRATCH_BYTES < _need(40, 1024, 6144, 16)
    s = lib.pbd_op_linear_static(40, 1024, 6144, 16, 2.0, None, None, 0x1000, 0x1000, None, None)
    assert s == 3  # PBD_ERR_CAPACITY, returned before the null pointers are even looked at
    msg = lib.pbd_op_last_error().decode()
    assert str(_need(40, 1024, 6144, 16)) in msg and str(SCRATCH_BYTES) in msg
    # a weight whose tiles alone exceed the scratch
    assert lib.pbd_op_linear_static(1, 4096, 4096, 0, 1.0, None, None, None, None, None, None) == 3
    # unsupported sizes and null pointers
    assert lib.pbd_op_linear_static(17, 1000, 128, 16, 2.0, None, None, None, None, None, None) == 1
    assert lib.pbd_op_linear_static(17, 1024, 100, 0, 2.0, None, None, None, None, None, None) == 1
    assert lib.pbd_op_linear_static(17, 1024, 128, 0, 2.0, None, None, None, None, None, None) == 1
    assert b"null pointer" in lib.pbd_op_last_error()


def _bf16(rng, shape, std):
    return synth.bf16_bits((rng.standard_normal(shape) * std).astype(np.float32))


def _dev(torch, bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


@pytest.mark.gpu
def test_static_scratch_matches_workspace_linear_on_consecutive_calls(lib):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    # call 1 fills most of the scratch (gate|up-shaped, rank 16); call 2 has another shape (fewer
    # rows, a longer K in more slices, rank 8), so its tiles and partial sums lie on bytes call 1
    # wrote: its result must not depend on them
    cases = [(17, 1024, 6144, 16, 11), (5, 3072, 1024, 8, 12)]
    inputs = []
    for M, K, N, r, seed in cases:
        rng = np.random.default_rng(seed)
        x = _dev(torch, _bf16(rng, (M, K), 1.0))
        W = _dev(torch, _bf16(rng, (N, K), 0.02))
        A = _dev(torch, _bf16(rng, (r, K), 0.02))
        B = _dev(torch, _bf16(rng, (N, r), 0.02))
        y = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
        inputs.append((x, W, A, B, y))
    torch.cuda.synchronize()
    before = torch.cuda.memory_allocated()
    # two calls in a row on the same stream, no synchronisation between them
    for x, W, A, B, y in inputs:
        pbd.pbd_op_linear_static(x, W, A, B, 2.0, y=y, sync=False)
    torch.cuda.synchronize()
    assert torch.cuda.memory_allocated() == before  # the calls took no memory from torch
    assert pbd.pbd_op_linear_static_status() == 0  # no kernel latched a device error
    for (x, W, A, B, y), (M, K, N, r, _) in zip(inputs, cases):
        ref = pbd.pbd_op_linear(x, W, A, B, 2.0).float().cpu().numpy()
        got = y.float().cpu().numpy()
        assert np.isfinite(got).all()
        # same tolerance as the linear's oracle test (two bf16 ulps of the magnitude) ...
        bad = np.abs(got - ref) > np.abs(ref) * 2.0 ** -7 + 1e-6
        assert not bad.any(), "M=%d K=%d N=%d r=%d: %d outputs differ" % (M, K, N, r, int(bad.sum()))
        # ... and, since both run the same kernels with the same fixed-order sums, identical
        assert np.array_equal(got, ref)
