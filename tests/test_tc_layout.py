"""Split-weight images of the tensor-core kernels (csrc/mca_tc_layout.h), checked on the CPU.

The header is plain C++; a probe compiled with g++ prints the offsets it assigns. They are compared
with the canonical K-major, no-swizzle operand layout of tcgen05 shared-memory matrix descriptors
(PTX ISA, "Shared memory matrix layout"): a core matrix is 8 rows x 16 bytes stored as 128
contiguous bytes; element (row n, column kk) of an operand read from start address S with leading
byte offset LBO (between core matrices adjacent in K) and stride byte offset SBO (between 8-row
groups) sits at S + (n // 8) * SBO + (kk // 4) * LBO + (n % 8) * 16 + (kk % 4) * 4.
"""
import os
import subprocess

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "paper_2607_08406_gb300", "csrc", "mca_tc_layout.h")

PROBE = r"""
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include "%s"
int main(int argc, char** argv) {
  if (!strcmp(argv[1], "idx")) {            // idx R rows cols: offsets of W[r][k], row-major
    const int R = atoi(argv[2]), rows = atoi(argv[3]), cols = atoi(argv[4]);
    printf("%%zu\n", mca::tc_image_lo(R));
    for (int r = 0; r < rows; ++r)
      for (int k = 0; k < cols; ++k) printf("%%zu\n", mca::tc_image_index(r, k, R, cols));
  } else if (!strcmp(argv[1], "tfm")) {     // tfm F nL: every matrix entry's hi and lo offsets
    const int F = atoi(argv[2]), nL = atoi(argv[3]);
    printf("%%zu %%zu\n", mca::tfm_tc_block_floats(F), mca::tfm_tc_image_floats(F, nL));
    for (int b = 0; b <= nL; ++b)
      for (int m = 0; m < 7; ++m) {
        if ((b == nL) != (m == mca::kTcHead)) continue;
        const int rows = m == mca::kTcW1 ? F : 128, cols = m == mca::kTcW2 ? F : 128;
        const size_t lo = mca::tc_image_lo(mca::tfm_tc_rows(m));
        for (int r = 0; r < rows; ++r)
          for (int k = 0; k < cols; ++k) {
            const size_t o = mca::tfm_tc_image_offset(m, b, r, k, F, nL);
            printf("%%d %%d %%d %%d %%zu %%zu\n", b, m, r, k, o, o + lo);
          }
      }
  } else {                                  // ok T d H F V B
    printf("%%d\n", (int)mca::tfm_tc_shape_ok(atoi(argv[2]), atoi(argv[3]), atoi(argv[4]),
                                             atoi(argv[5]), atoi(argv[6]), atoll(argv[7])));
  }
  return 0;
}
"""


@pytest.fixture(scope="module")
def probe(tmp_path_factory):
    d = tmp_path_factory.mktemp("tclayout")
    src = d / "probe.cpp"
    src.write_text(PROBE % HEADER)
    exe = d / "probe"
    subprocess.run(["g++", "-std=c++17", "-O1", str(src), "-o", str(exe)], check=True)

    def run(*args):
        out = subprocess.run([str(exe), *map(str, args)], check=True, capture_output=True,
                             text=True).stdout
        return out.split("\n")[:-1]

    return run


def image(probe, R, rows, cols):
    lines = probe("idx", R, rows, cols)
    lo = int(lines[0])
    return lo, np.array([int(x) for x in lines[1:]], dtype=np.int64).reshape(rows, cols)


@pytest.mark.parametrize("R,rows,cols", [(128, 128, 128), (64, 512, 128), (128, 128, 512),
                                         (256, 256, 256), (64, 128, 64)])
def test_image_matches_descriptor_layout(probe, R, rows, cols):
    """Every chunk (R rows x 16 columns) read through descriptors with LBO = 16 R, SBO = 128 at
    start = chunk + 2 LBO ks (hi) and + 4 LBO more (lo) yields exactly W[r][k]."""
    lo, off = image(probe, R, rows, cols)
    lbo, sbo = 16 * R, 128
    assert lo * 4 == 4 * lbo
    allb = []
    for rb in range(rows // R):
        for kc in range(cols // 16):
            chunk = (rb * (cols // 16) + kc) * R * 32 * 4          # bytes
            for ks in range(2):
                start = chunk + ks * 2 * lbo
                n = np.arange(R)[:, None]
                kk = np.arange(8)[None, :]
                want = start + (n // 8) * sbo + (kk // 4) * lbo + (n % 8) * 16 + (kk % 4) * 4
                got = 4 * off[rb * R + n, kc * 16 + ks * 8 + kk]
                np.testing.assert_array_equal(got, want)
                allb.append(got.ravel())
    # hi and lo parts together tile the image exactly once
    hi = np.concatenate(allb) // 4
    both = np.sort(np.concatenate([hi, hi + lo]))
    np.testing.assert_array_equal(both, np.arange(2 * rows * cols))


def test_transformer_images_tile_and_follow_the_chunk_order(probe):
    """Per block: Wq Wk Wv Wo as 8 chunks of 4096 floats each (32 in a row), W1 as (hidden pair p,
    K chunk u) 4096-float chunks from 131072, W2 as 4096-float chunks from 131072 + 256 F; the head
    after the last block. Hi and lo offsets of all entries tile the image exactly once."""
    F, nL = 128, 2
    lines = probe("tfm", F, nL)
    blk, total = map(int, lines[0].split())
    assert blk == 4 * 32768 + 512 * F and total == nL * blk + 32768
    a = np.array([list(map(int, x.split())) for x in lines[1:]], dtype=np.int64)
    b, m, r, k, hi, lo = a.T
    np.testing.assert_array_equal(np.sort(np.concatenate([hi, lo])), np.arange(total))
    base = np.where(m == 6, nL * blk, b * blk)
    # the chunk each entry lies in, as the kernels' loader addresses chunks
    qkvo = m <= 3
    start = np.empty_like(hi)
    size = np.empty_like(hi)
    start[qkvo] = base[qkvo] + (m[qkvo] * 8 + k[qkvo] // 16) * 4096
    size[qkvo] = 4096
    w1 = m == 4
    start[w1] = base[w1] + 131072 + ((r[w1] // 128) * 8 + k[w1] // 16) * 4096
    size[w1] = 4096
    w2 = m == 5
    start[w2] = base[w2] + 131072 + 256 * F + (k[w2] // 16) * 4096
    size[w2] = 4096
    hd = m == 6
    start[hd] = base[hd] + (k[hd] // 16) * 4096
    size[hd] = 4096
    for part in (hi, lo):
        assert np.all(part >= start) and np.all(part < start + size)


def test_shape_gate(probe):
    """The character-level workload (T 64, d 128, 4 heads, FFN 512, vocabulary 65, 256 sequences)
    qualifies; other widths, an FFN that is not a multiple of 128 (W1 is issued 128 hidden units at
    a time), odd sequence counts, or a vocabulary above 128 do not."""
    assert probe("ok", 64, 128, 4, 512, 65, 256) == ["1"]
    assert probe("ok", 64, 128, 4, 128, 65, 2) == ["1"]
    for args in [(32, 128, 4, 512, 65, 256), (64, 96, 4, 512, 65, 256), (64, 128, 2, 512, 65, 256),
                 (64, 128, 4, 500, 65, 256), (64, 128, 4, 192, 65, 256), (64, 128, 4, 64, 65, 256),
                 (64, 128, 4, 512, 200, 256), (64, 128, 4, 512, 65, 255)]:
        assert probe("ok", *args) == ["0"], args
