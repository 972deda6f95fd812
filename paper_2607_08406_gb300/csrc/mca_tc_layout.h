// Split-weight images read by the tensor-core kernels (host and device; plain C++ without CUDA).
//
// A kind::tf32 MMA reads a weight matrix W [rows x cols] as its B operand (N = rows, K = cols),
// K-major without swizzle: core matrices of 8 rows x 4 tf32 (16 bytes a row, 128 contiguous
// bytes). Each weight is kept split, W = W_hi + W_lo with both parts rounded to tf32, so that three
// tf32 MMAs give an fp32-accurate product (3xTF32). The rows are cut into blocks of R rows, each
// block's columns into chunks of 16; one chunk is one bulk copy of R * 128 bytes:
//   the high parts of its four 4-column groups (R rows x 16 bytes each, so the descriptor's
//   K-direction core-matrix stride is R * 16 bytes and its 8-row stride 128 bytes), then the low
//   parts in the same order (R * 16 floats further on).
#pragma once

#include <cstddef>

#if defined(__CUDACC__)
#define MCA_HD __host__ __device__ __forceinline__
#else
#define MCA_HD inline
#endif

namespace mca {

// Float offset of the high part of W[r][k] (R divides rows and is a multiple of 8; cols is a
// multiple of 16).
MCA_HD size_t tc_image_index(int r, int k, int R, int cols) {
  return ((size_t)(r / R) * (size_t)(cols >> 4) + (size_t)(k >> 4)) * (size_t)R * 32 +
         (size_t)((k >> 2) & 3) * (size_t)R * 4 + (size_t)(r % R) * 4 + (size_t)(k & 3);
}

// Distance in floats from a high part to its low part.
MCA_HD size_t tc_image_lo(int R) { return (size_t)R * 16; }

// Transformer (d_model 128, d_ff = F a multiple of 128): per block Wq, Wk, Wv, Wo (128 x 128,
// R = 128), W1 (F x 128, R = 128: the hidden units of two 64-wide FFN chunks per row block), W2
// (128 x F, R = 128); after the last block the head (vocab rows, padded with zero rows to 128,
// R = 128).
enum TfmTcMat { kTcMatNone = -1, kTcQ = 0, kTcK = 1, kTcV = 2, kTcO = 3, kTcW1 = 4, kTcW2 = 5,
                kTcHead = 6 };

constexpr int kTcTfmD = 128;        // model width of the tensor-core Transformer kernels
constexpr int kTcTfmT = 64;         // tokens per sequence
constexpr int kTcTfmHeads = 4;
constexpr int kTcTfmHc = 64;        // feed-forward hidden columns per chunk (activation, W2)
constexpr int kTcTfmHp = 128;       // feed-forward hidden columns per W1 product (two chunks)

MCA_HD size_t tfm_tc_block_floats(int F) { return (size_t)4 * 32768 + (size_t)512 * F; }
MCA_HD size_t tfm_tc_image_floats(int F, int nL) {
  return (size_t)nL * tfm_tc_block_floats(F) + 32768;
}
MCA_HD int tfm_tc_rows(int) { return 128; }

// Float offset of the high part of element (r, k) of matrix `mat` of block b.
MCA_HD size_t tfm_tc_image_offset(int mat, int b, int r, int k, int F, int nL) {
  const size_t blk = tfm_tc_block_floats(F);
  if (mat == kTcHead) return (size_t)nL * blk + tc_image_index(r, k, 128, kTcTfmD);
  const size_t base = (size_t)b * blk;
  if (mat <= kTcO) return base + (size_t)mat * 32768 + tc_image_index(r, k, 128, kTcTfmD);
  if (mat == kTcW1) return base + 131072 + tc_image_index(r, k, kTcTfmHp, kTcTfmD);
  return base + 131072 + (size_t)256 * F + tc_image_index(r, k, 128, F);
}

// Shapes the tensor-core Transformer kernels handle: T = 64, d = 128, 4 heads of 32, d_ff a
// multiple of 128 up to 1024, vocab <= 128, an even number of sequences (two per CTA).
MCA_HD bool tfm_tc_shape_ok(int T, int d, int H, int F, int V, long long B) {
  return T == kTcTfmT && d == kTcTfmD && H == kTcTfmHeads && F % kTcTfmHp == 0 && F >= kTcTfmHp &&
         F <= 1024 && V >= 2 && V <= 128 && B % 2 == 0;
}

}  // namespace mca
