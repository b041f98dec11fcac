"""GPU parity of the prefill's tensor-core matrix product (kfl_matmul_bf16w: fp32 activations as
two bf16 terms, bf16 weights) against the fp64 product of the same values.

Bar: every element within 1e-4 of the row's fp64 RMS plus 2^-14 relative (x carried to about 2^-16
relative by its two terms, fp32 accumulation over K <= 4096 products; the sums' order is the
kernel's).  Shapes span several 128 x 256 output tiles, K tiles of 128 and their 64-column halves,
with ragged tails on T, N and K.
"""
import numpy as np
import pytest
import torch

from gpu_helpers import ensure_built
from paper_2609_34045_gb300 import stage as K

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    ensure_built()
    torch.cuda.init()


@pytest.mark.parametrize("T,Kd,N", [(128, 64, 256), (300, 320, 700), (1, 128, 1000), (257, 1000, 513),
                                    (128, 4096, 256), (640, 3584, 1152)])
def test_matmul_matches_fp64(T, Kd, N):
    rng = np.random.default_rng(T * 7919 + Kd * 31 + N)
    x = rng.standard_normal((T, Kd)).astype(np.float32)
    w = torch.from_numpy((rng.standard_normal((N, Kd)) * 0.05).astype(np.float32)).to(torch.bfloat16)
    ldx = Kd + 3
    xd = torch.zeros(T, ldx, dtype=torch.float32, device="cuda")
    xd[:, :Kd] = torch.from_numpy(x).cuda()
    ldy = (N + 3) // 4 * 4 + 4
    y = torch.full((T, ldy), 7.0, dtype=torch.float32, device="cuda")
    K.kfl_matmul_bf16w(xd, T, Kd, ldx, w.view(torch.int16).cuda().contiguous(), N, y, ldy,
                       torch.cuda.current_stream().cuda_stream)
    got = y.cpu().numpy()
    ref = x.astype(np.float64) @ w.to(torch.float64).numpy().T
    rms = np.sqrt(np.mean(ref * ref, axis=1, keepdims=True))
    err = np.abs(got[:, :N] - ref)
    assert np.all(err <= 1e-4 * rms + 2.0 ** -14 * np.abs(ref)), float(np.max(err / rms))
    assert np.all(got[:, N:] == 7.0)  # columns past N untouched


def test_matmul_argument_errors():
    x = torch.zeros(4, 64, dtype=torch.float32, device="cuda")
    w = torch.zeros(8, 64, dtype=torch.int16, device="cuda")
    y = torch.zeros(4, 8, dtype=torch.float32, device="cuda")
    with pytest.raises(K.KflError):
        K.kfl_matmul_bf16w(x, 4, 64, 60, w, 8, y, 8)   # ldx < K
    with pytest.raises(K.KflError):
        K.kfl_matmul_bf16w(x, 4, 64, 64, w, 8, y, 6)   # ldy < N
    with pytest.raises(K.KflError):
        K.kfl_matmul_bf16w(x, 0, 64, 64, w, 8, y, 8)
