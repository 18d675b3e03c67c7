"""The learners' dense product (auv_gemm: the contractions of the PPO update
and the SHAC window, paper §III-A) through the C ABI against a float64
product of the same operands, for every operand layout the learners use:

- forward   C[b][h] = sum_k X[b][k] W[h][k]        (A, B K-major)
- input grad C[b][i] = sum_h G[b][h] W[h][i]       (B MN-major: W read by column)
- weight grad C[h][i] = sum_b G[b][h] H[b][i]      (A, B MN-major; K = the
  batch, split over CTAs and added in a fixed order)

Tolerances, as a fraction of sum_k |A(m,k) B(n,k)| for each output:
- bf16: products of bf16 operands are exact in fp32, the fp32 sums carry a
  relative rounding error of a few 2^-24 per addition: 1e-5;
- tf32: each fp32 operand enters the product with its low 13 mantissa bits
  dropped (relative error below 2^-10 each), so a product is off by at most
  about 2^-9: 3e-3;
- fp32 (CUDA cores): fp32 products and sums: 1e-5.
bf16 outputs add half a bf16 ulp (2^-9 relative) of the result."""
import numpy as np
import pytest

from parity_util import need_gpu

pytestmark = pytest.mark.gpu

TOL = {"bf16": 1e-5, "tf32": 3e-3, "fp32": 1e-5}


def _operand(torch, rng, rows, k, mn, dtype, ld_pad=0, ld_mult=1):
    """A random operand with element (r, k) at r*ld + k (mn False) or k*ld + r;
    ld = inner size + ld_pad, rounded up to a multiple of ld_mult."""
    inner = rows if mn else k
    outer = k if mn else rows
    ld = -(-(inner + ld_pad) // ld_mult) * ld_mult
    full = rng.standard_normal((outer, ld)).astype(np.float32)
    t = torch.from_numpy(full).cuda().to(dtype).contiguous()
    vals = t.float().cpu().numpy().astype(np.float64)[:, :inner]
    logical = vals.T if mn else vals           # [rows][k]
    return t, ld, logical


CASES = [
    # precision, M, N, K, a_mn, b_mn, c_bf16, beta, ld_pad
    ("bf16", 1000, 256, 24, False, False, False, 0.0, 0),       # layer 1 forward (Dp = 24)
    ("bf16", 777, 264, 264, False, False, True, 0.0, 0),        # layer 2 forward, bf16 out
    ("bf16", 1000, 256, 16, False, True, True, 0.0, 0),         # gH2 = gY W3 (K = 16)
    ("bf16", 2000, 264, 256, False, True, False, 1.0, 8),       # gH1 = gZ2 W2, accumulate
    ("bf16", 256, 264, 65536, True, True, False, 0.0, 8),       # gW2, split over the batch
    ("bf16", 16, 264, 5000, True, True, False, 1.0, 0),         # gW3 (out = 16), ragged K
    ("bf16", 256, 24, 9999, True, True, False, 0.0, 0),         # gW1 (Dp = 24)
    ("bf16", 1, 1, 1, False, False, False, 0.0, 7),             # smallest
    ("bf16", 500, 300, 64, False, False, False, 0.0, 0),        # 320-wide tile, K-major B
    ("bf16", 300, 290, 3000, True, True, True, 1.0, 0),         # 320-wide tile, bf16 out
    ("tf32", 1000, 256, 24, False, False, False, 0.0, 0),
    ("tf32", 4096, 264, 264, False, False, False, 0.0, 0),
    ("tf32", 1000, 256, 264, False, True, False, 0.0, 0),
    ("tf32", 256, 264, 32768, True, True, False, 1.0, 4),
    ("tf32", 16, 264, 3000, True, True, False, 0.0, 0),
    ("tf32", 3, 5, 7, True, False, False, 0.0, 1),
    ("tf32", 500, 290, 40, False, False, False, 0.0, 0),        # 320-wide tile
    ("fp32", 1000, 256, 24, False, False, False, 0.0, 0),
    ("fp32", 513, 264, 256, False, True, False, 1.0, 3),
    ("fp32", 256, 264, 20000, True, True, False, 0.0, 0),
    ("fp32", 2, 3, 1, True, True, False, 0.0, 0),
    ("fp32", 16, 264, 5000, True, True, False, 1.0, 0),         # 32-row tile: gW3
    ("fp32", 1, 264, 3001, True, True, False, 0.0, 2),          # value head gW3 (out = 1)
    ("fp32", 32, 130, 77, False, True, False, 0.0, 1),          # 32-row tile, K-major A
    ("fp32", 33, 129, 40, True, False, False, 1.0, 0),          # just over: 128-row tile
]


@pytest.mark.parametrize("prec,M,N,K,a_mn,b_mn,c_bf16,beta,pad", CASES)
def test_gemm_against_float64(prec, M, N, K, a_mn, b_mn, c_bf16, beta, pad):
    torch = need_gpu()
    from paper_2512_13359_gb300 import auvenv
    rng = np.random.default_rng(M * 7919 + N * 31 + K)
    dt = torch.bfloat16 if prec == "bf16" else torch.float32
    # tensor-core operands: ld * element size a multiple of 16 bytes
    mult = {"bf16": 8, "tf32": 4, "fp32": 1}[prec]
    A, lda, a_log = _operand(torch, rng, M, K, a_mn, dt, pad, mult)
    B, ldb, b_log = _operand(torch, rng, N, K, b_mn, dt, pad, mult)
    ldc = N + 5
    cdt = torch.bfloat16 if c_bf16 else torch.float32
    C0 = torch.from_numpy(rng.standard_normal((M, ldc)).astype(np.float32)).cuda().to(cdt)
    Cout = C0.clone()
    ws = torch.empty(max(1, auvenv.lib().auv_gemm_workspace_bytes(M, N, K)) // 4 + 1,
                     dtype=torch.float32, device="cuda")
    st = auvenv.gemm(prec, M, N, K, A, lda, a_mn, B, ldb, b_mn, Cout, ldc, beta, ws)
    torch.cuda.synchronize()
    assert st.cpu().tolist() == [0, 0, 0, 0]
    ref = a_log @ b_log.T
    scale = np.abs(a_log) @ np.abs(b_log).T
    c0 = C0.float().cpu().numpy().astype(np.float64)
    ref = ref + beta * c0[:, :N]
    got = Cout.float().cpu().numpy().astype(np.float64)
    tol = TOL[prec] * scale + 1e-30
    if c_bf16:
        tol = tol + 2.0 ** -8 * np.abs(ref) + (np.abs(c0[:, :N]) * 2.0 ** -8 if beta else 0.0)
    err = np.abs(got[:, :N] - ref)
    print(f"[gemm {prec} {M}x{N}x{K} a_mn={a_mn} b_mn={b_mn}] max err / scale "
          f"{(err / np.maximum(scale, 1e-30)).max():.2e}")
    assert np.all(err <= tol), f"max excess {(err - tol).max():.3e}"
    # columns beyond N untouched
    assert torch.equal(Cout[:, N:], C0[:, N:])


@pytest.mark.parametrize("prec,M,N,K,c_bf16", [
    ("bf16", 1000, 256, 24, False), ("bf16", 777, 264, 264, True), ("tf32", 513, 256, 40, False),
    ("bf16", 300, 290, 64, True)])
def test_gemm_sector_aligned_output(prec, M, N, K, c_bf16):
    """C rows on 32-byte boundaries (ldc a multiple of 16): the epilogue's
    whole-sector stores; the columns past N stay untouched."""
    torch = need_gpu()
    from paper_2512_13359_gb300 import auvenv
    rng = np.random.default_rng(M + N + K)
    dt = torch.bfloat16 if prec == "bf16" else torch.float32
    mult = {"bf16": 8, "tf32": 4}[prec]
    A, lda, a_log = _operand(torch, rng, M, K, False, dt, 0, mult)
    B, ldb, b_log = _operand(torch, rng, N, K, False, dt, 0, mult)
    ldc = -(-N // 16) * 16 + 16
    cdt = torch.bfloat16 if c_bf16 else torch.float32
    C0 = torch.from_numpy(rng.standard_normal((M, ldc)).astype(np.float32)).cuda().to(cdt)
    Cout = C0.clone()
    ws = torch.empty(max(1, auvenv.lib().auv_gemm_workspace_bytes(M, N, K)) // 4 + 1,
                     dtype=torch.float32, device="cuda")
    st = auvenv.gemm(prec, M, N, K, A, lda, False, B, ldb, False, Cout, ldc, 0.0, ws)
    torch.cuda.synchronize()
    assert st.cpu().tolist() == [0, 0, 0, 0]
    ref = a_log @ b_log.T
    scale = np.abs(a_log) @ np.abs(b_log).T
    got = Cout.float().cpu().numpy().astype(np.float64)[:, :N]
    tol = TOL[prec] * scale + 1e-30 + (2.0 ** -8 * np.abs(ref) if c_bf16 else 0.0)
    assert np.all(np.abs(got - ref) <= tol)
    assert torch.equal(Cout[:, N:], C0[:, N:])


def test_gemm_rejects_bad_operands():
    torch = need_gpu()
    from paper_2512_13359_gb300 import auvenv
    A = torch.zeros(64 * 40 + 8, dtype=torch.bfloat16, device="cuda")
    Cm = torch.zeros((64, 40), device="cuda")
    with pytest.raises(auvenv.AuvError) as e:          # misaligned operand for TMA
        auvenv.gemm("bf16", 64, 40, 40, A[1:], 40, False, A, 40, False, Cm, 40)
    assert e.value.code == auvenv.AUV_ERR_SIZE
    with pytest.raises(auvenv.AuvError) as e:          # ld * 2 bytes not a multiple of 16
        auvenv.gemm("bf16", 64, 40, 36, A, 36, False, A, 40, False, Cm, 40)
    assert e.value.code == auvenv.AUV_ERR_SIZE
    with pytest.raises(auvenv.AuvError) as e:          # ldc < N
        auvenv.gemm("bf16", 64, 40, 40, A, 40, False, A, 40, False, Cm, 39)
    assert e.value.code == auvenv.AUV_ERR_INVALID
