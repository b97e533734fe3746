"""Per-kernel parity on the GPU: the tensor-core linear (+ adapter delta) and the lm_head argmax
against the CPU oracle's steps, element by element, at shapes that span several tiles, ragged
token counts and every K split used by the passes."""
import ctypes as C

import numpy as np
import pytest

from oracle import model as om
from paper_2607_12422_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch_dev():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_12422_gb300 import pbd
    pbd.load()
    return torch


def _bf16(rng, shape, std):
    return synth.bf16_bits((rng.standard_normal(shape) * std).astype(np.float32))


def _to_dev(torch, bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def _oracle_linear(shape, x_bits, W, A, B, on):
    x = synth.bf16_to_f32(x_bits)
    M, K = x.shape
    N = W.shape[0]
    y = np.empty((M, N), np.float32)
    cfg = om.make_config(shape)
    om.lib().orc_op_linear(C.byref(cfg), M, K, N, om._fp(np.ascontiguousarray(x)), om._u16(W),
                           om._u16(A), om._u16(B), int(on), om._fp(y))
    return y


class _Shape:
    def __init__(self, r, scale):
        self.n_layers, self.hidden, self.n_q_heads, self.n_kv_heads = 1, 128, 1, 1
        self.head_dim, self.intermediate, self.vocab = 128, 128, 128
        self.rms_eps, self.rope_theta, self.lora_rank, self.lora_alpha = 1e-6, 1e6, r, scale * r


@pytest.mark.parametrize("M,K,N,r", [(1, 1024, 128, 16), (17, 1024, 4096, 16), (17, 2048, 1024, 16),
                                     (17, 3072, 1024, 16), (33, 256, 768, 8), (136, 1024, 6144, 16),
                                     (300, 512, 384, 0), (5, 768, 256, 8)])
def test_linear_matches_oracle(torch_dev, M, K, N, r):
    from paper_2607_12422_gb300 import pbd
    torch = torch_dev
    rng = np.random.default_rng(M * 7 + K + N)
    x = _bf16(rng, (M, K), 1.0)
    W = _bf16(rng, (N, K), 0.02)
    A = _bf16(rng, (max(r, 1), K), 0.02)
    B = _bf16(rng, (N, max(r, 1)), 0.02)
    scale = 2.0
    y = pbd.pbd_op_linear(_to_dev(torch, x), _to_dev(torch, W), _to_dev(torch, A) if r else None,
                          _to_dev(torch, B) if r else None, scale)
    got = y.float().cpu().numpy()
    ref = _oracle_linear(_Shape(max(r, 1), scale), x, W, A, B, r > 0)
    # both sides round an fp32 sum to bf16: allow two bf16 ulps of the magnitude
    tol = np.abs(ref) * 2.0 ** -7 + 1e-6
    bad = np.abs(got - ref) > tol
    assert not bad.any(), "max rel err %.3g at %s" % (
        float((np.abs(got - ref) / (np.abs(ref) + 1e-6)).max()), np.argwhere(bad)[:5].tolist())
    # most outputs agree exactly (same rounding of nearly the same fp32 sum)
    assert (got == ref).mean() > 0.95


@pytest.mark.parametrize("M,H,V", [(1, 1024, 4096), (17, 1024, 18944), (16, 256, 4096), (136, 1024, 2048),
                                   (200, 256, 1024)])
def test_lm_head_argmax_matches_oracle(torch_dev, M, H, V):
    from paper_2607_12422_gb300 import pbd
    torch = torch_dev
    rng = np.random.default_rng(M + H + V)
    x = _bf16(rng, (M, H), 1.0)
    E = _bf16(rng, (V, H), 0.02)
    ids, lg = pbd.pbd_op_lm_head_argmax(_to_dev(torch, x), _to_dev(torch, E), want_logits=True)
    ref = synth.bf16_to_f32(x).astype(np.float64) @ synth.bf16_to_f32(E).astype(np.float64).T
    got = lg.cpu().numpy()
    assert np.abs(got - ref).max() < 1e-4 * (1 + np.abs(ref).max())
    ids = ids.cpu().numpy()
    for m in range(M):
        # exact argmax of the GPU's own logits, lowest index on ties
        assert ids[m] == int(np.argmax(got[m]))
        srt = np.sort(ref[m])
        if srt[-1] - srt[-2] > 1e-4:
            assert ids[m] == int(np.argmax(ref[m]))


def test_op_status_reports_a_latched_device_code(torch_dev):
    """pbd_op_status maps the workspace's status word to PBD_ERR_DEVICE with the code (a word set
    here by hand: no kernel is made to fail), leaves a clean word PBD_OK, and a real call's word
    is clean."""
    torch = torch_dev
    from paper_2607_12422_gb300 import pbd
    L = pbd.load()
    buf = torch.zeros(4096, dtype=torch.uint8, device="cuda")
    off = (-buf.data_ptr()) % 1024
    ws = buf[off:off + 1024]
    st = torch.cuda.current_stream().cuda_stream
    code = C.c_int32(-1)
    assert L.pbd_op_status(ws.data_ptr(), st, C.byref(code)) == 0 and code.value == 0
    ws.view(torch.int32)[0] = 6  # DEV_TIMEOUT_DEP
    assert L.pbd_op_status(ws.data_ptr(), st, C.byref(code)) == 6 and code.value == 6
    assert b"device status 6" in L.pbd_op_last_error()
    # a real call: its own status word starts clean and stays clean
    rng = np.random.default_rng(3)
    x = _to_dev(torch, _bf16(rng, (5, 256), 1.0))
    W = _to_dev(torch, _bf16(rng, (128, 256), 0.02))
    y = pbd.pbd_op_linear(x, W)  # raises on a latched code
    assert y.shape == (5, 128)
    ids, _ = pbd.pbd_op_lm_head_argmax(x, W)
    assert ids.shape == (5,)
