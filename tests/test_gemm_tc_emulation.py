"""CPU emulation of the tensor-core forward GEMM's data movement (csrc/mca_gemm_tc.cu).

Test infrastructure, not the kernel: it repeats the kernel's arithmetic step by step -- the two
operand-image kernels (tc_image_index with R = 128 samples / 256 rows, K chunks of 16, hi then lo),
each stage's two bulk copies into a byte-addressed shared-memory array, every MMA executed from its
decoded descriptors under the canonical K-major no-swizzle layout (core matrices of 8 rows x 16
bytes; LBO between K-adjacent core matrices, SBO between 8-row groups) with tf32 operands, the
tensor-memory accumulator, and the epilogue's stores -- and compares the fields with a float64
product. A wrong stride, chunk offset, K step, hi/lo offset or epilogue index fails here; the
hardware, races and the compiled code are not covered.
"""
import numpy as np
import pytest

from tc_emulator import tc_image_index, tf32_rna, tf32_trunc, umma_desc, idesc

GM, GN, GK = 128, 256, 16
A_HALF, B_HALF = GM * GK * 4, GN * GK * 4
A_CHUNK, B_CHUNK = 2 * A_HALF, 2 * B_HALF
STAGE, STAGES = A_CHUNK + B_CHUNK, 2
ALBO, ASBO = (GM // 8) * 128, 128
BLBO, BSBO = (GN // 8) * 128, 128


def act(name, z):
    if name == "identity":
        return z
    if name == "tanh":
        return np.tanh(z)
    if name == "gaussian":
        return np.exp(-z * z)
    raise ValueError(name)


def act_image(B, K, Kp, Np, act_name):
    """act_image_kernel: thread (n, k0) writes 4 hi and 4 lo values."""
    img = np.zeros((Np // GM) * (Kp // GK) * (A_CHUNK // 4), np.float32)
    for k0 in range(0, Kp, 4):
        for q in range(4):
            k = k0 + q
            v = np.zeros(Np, np.float32)
            if k < K:
                v = B[k].astype(np.float32)
                if act_name is not None:
                    v = act(act_name, v.astype(np.float64)).astype(np.float32)
            hi = tf32_rna(v)
            lo = tf32_rna(v - hi)
            n = np.arange(Np)
            o = np.array([tc_image_index(int(x), k0, GM, Kp) for x in n]) + q
            img[o] = hi
            img[o + GM * 16] = lo
    return img


def w_image(W, M, K, Kp):
    img = np.zeros((M // GN) * (Kp // GK) * (B_CHUNK // 4), np.float32)
    for r in range(M):
        for k0 in range(0, Kp, 4):
            o = tc_image_index(r, k0, GN, Kp)
            for q in range(4):
                k = k0 + q
                v = np.float32(W[r, k]) if k < K else np.float32(0.0)
                hi = tf32_rna(v)
                img[o + q] = hi
                img[o + q + GN * 16] = tf32_rna(np.float32(v - hi))
    return img


def gather(sm, desc, rows):
    start = (desc & 0x3FFF) << 4
    lbo = ((desc >> 16) & 0x3FFF) << 4
    sbo = ((desc >> 32) & 0x3FFF) << 4
    n = np.arange(rows)[:, None]
    k = np.arange(8)[None, :]
    addr = start + (n // 8) * sbo + (k // 4) * lbo + (n % 8) * 16 + (k % 4) * 4
    assert np.all(addr % 4 == 0)
    return tf32_trunc(sm[addr // 4])


def run_cta(aimg, bimg, nch, bs, bf, Z, Np):
    sm = np.zeros(STAGES * STAGE // 4, np.float32)
    tm = np.zeros((GM, GN), np.float32)
    ag = bs * nch * (A_CHUNK // 4)
    bg = bf * nch * (B_CHUNK // 4)
    idsc = idesc(GM, GN)
    assert ((idsc >> 17) & 0x3F) << 3 == GN and ((idsc >> 24) & 0x1F) << 4 == GM
    for c in range(nch):
        st = c % STAGES
        base = st * STAGE // 4
        sm[base:base + A_CHUNK // 4] = aimg[ag + c * (A_CHUNK // 4):ag + (c + 1) * (A_CHUNK // 4)]
        sm[base + A_CHUNK // 4:base + STAGE // 4] = \
            bimg[bg + c * (B_CHUNK // 4):bg + (c + 1) * (B_CHUNK // 4)]
        sa, sb = st * STAGE, st * STAGE + A_CHUNK
        for ks in range(GK // 8):
            ahi = umma_desc(sa + ks * 2 * ALBO, ALBO, ASBO)
            alo = umma_desc(sa + A_HALF + ks * 2 * ALBO, ALBO, ASBO)
            bhi = umma_desc(sb + ks * 2 * BLBO, BLBO, BSBO)
            blo = umma_desc(sb + B_HALF + ks * 2 * BLBO, BLBO, BSBO)
            for a_d, b_d, first in ((alo, bhi, True), (ahi, blo, False), (ahi, bhi, False)):
                D = (gather(sm, a_d, GM).astype(np.float64)
                     @ gather(sm, b_d, GN).astype(np.float64).T).astype(np.float32)
                if first and c == 0 and ks == 0:
                    tm[:] = D
                else:
                    tm[:] = (tm.astype(np.float64) + D).astype(np.float32)
    # epilogue: warp w, lane -> sample row 32 w + lane; 16 columns per tensor-memory load
    for w in range(4):
        for lane in range(32):
            n = bs * GM + w * 32 + lane
            for c0 in range(0, GN, 16):
                for q in range(16):
                    Z[(bf * GN + c0 + q) * Np + n] = tm[w * 32 + lane, c0 + q]


@pytest.mark.parametrize("M,K,Np,act_name", [(256, 40, 128, "tanh"), (512, 32, 256, None),
                                             (256, 24, 128, "gaussian")])
def test_gemm_tc_emulation_matches_float64_product(M, K, Np, act_name):
    rng = np.random.default_rng(M + K)
    W = rng.uniform(-0.5, 0.5, (M, K)).astype(np.float32)
    B = rng.uniform(-1.5, 1.5, (K, Np)).astype(np.float32)
    Kp = (K + GK - 1) // GK * GK
    nch = Kp // GK
    aimg = act_image(B, K, Kp, Np, act_name)
    bimg = w_image(W, M, K, Kp)
    Z = np.full(M * Np, np.nan, np.float32)
    for bs in range(Np // GM):
        for bf in range(M // GN):
            run_cta(aimg, bimg, nch, bs, bf, Z, Np)
    Z = Z.reshape(M, Np)
    A = B.astype(np.float64) if act_name is None else act(act_name, B.astype(np.float64))
    want = W.astype(np.float64) @ A
    assert np.all(np.isfinite(Z))
    scale = np.abs(W.astype(np.float64)) @ np.abs(A)
    assert np.max(np.abs(Z - want) / scale) < 2e-6


def test_gemm_tc_emulation_exact_on_dyadic_operands():
    """Dyadic operands (k / 256 inputs, q / 512 weights) are exact in tf32: the lo parts are 0 and
    every partial sum is exact, so the fields equal the exact product bit for bit."""
    rng = np.random.default_rng(5)
    M, K, Np = 256, 48, 128
    W = (rng.integers(-64, 65, (M, K)) / 512.0).astype(np.float32)
    B = (rng.integers(0, 256, (K, Np)) / 256.0).astype(np.float32)
    Kp = K
    aimg = act_image(B, K, Kp, Np, None)
    bimg = w_image(W, M, K, Kp)
    Z = np.zeros(M * Np, np.float32)
    run_cta(aimg, bimg, Kp // GK, 0, 0, Z, Np)
    want = (W.astype(np.float64) @ B.astype(np.float64)).astype(np.float32)
    assert np.array_equal(Z.reshape(M, Np), want)
