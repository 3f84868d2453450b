// mc_layout.h -- the packed expert-weight layout (private to the library) and the
// offset tables the expert kernels use.  Host and device code include it.
//
// Storage of one quantised matrix W [R, K] (groups of g along K, b bits):
//   tile      = 16 rows x 128 columns; bytes = 256*b (codes) + 64*(128/g) (meta)
//   supertile = the 8 tiles of a 128-row block at one 128-column step (STB bytes)
// Supertiles are stored so that the expert kernels stream one large contiguous
// block per step:
//   W1 / W3 of an expert share one region, interleaved per supertile:
//       [F/128 row blocks][H/128 column steps][W1 supertile][W3 supertile]
//   W2 pairs its row blocks:
//       [H/256 row-block pairs][F/128 column steps][block 2p][block 2p+1]
//       (when H/128 is odd the last pair holds one block)
// Inside a tile every one of the 32 lanes of a warp owns 64 codes: rows r0 = g8
// and r1 = g8 + 8 (g8 = lane / 4), and for each row two runs of 16 consecutive
// columns, so that an mma.sync.m16n8k16 A-fragment register (two consecutive
// columns of one row) comes out of the packed word with a single AND/OR.
//   pair j (0..31) of lane (g8, t):  step s = j/4, rho = j%4
//       row  = g8 + 8*(rho & 1)
//       col  = 64*(s/4) + 16*t + 4*(s%4) + 2*(rho >> 1)   (and col + 1)
// The k-step s of the mma therefore only touches columns of one 64-column half,
// so groups of 64 and of 128 are both whole k-steps.
//
// Code words of a lane (b = bits):
//   2-bit field plane, 4 words: word i holds pairs 8i..8i+7; pair position
//       p = j%8 has its low-column code at bits [2p, 2p+1] and its high-column
//       code at bits [16+2p, 17+2p].
//   1-bit field plane, 2 words: word i holds pairs 16i..16i+15; position
//       p = j%16 at bit p (low column) and bit 16+p (high column).
//   b = 1: one 1-bit plane;  b = 2: one 2-bit plane;
//   b = 3: a 2-bit plane of q & 3 followed by a 1-bit plane of q >> 2.
// Code bytes of a tile: plane-major, then lane-major (lane l's words contiguous):
//   [2-bit plane: 32 lanes x 16 B][1-bit plane: 32 lanes x 8 B] (as present).
// Meta bytes of a tile: [group-in-tile][g8 = 0..7][s(r0), z(r0), s(r1), z(r1)] fp16.
//
// Decoding without shifts per field: a field at mantissa position p' of an fp16
// whose exponent field is set to 15 + E reads as 2^E + q * 2^(E + width*p' - 10);
// choosing E = 10 - width*p' makes it (2^E + q).  The constant 2^E ("offset")
// depends only on the field position, so sum_k (off_k + q_k) x_k - sum_k off_k x_k
// = sum_k q_k x_k, and the second sum is a per-(vector, group) table.
#pragma once
#include <stdint.h>

#if defined(__CUDACC__)
#define MC_HD __host__ __device__ __forceinline__
#else
#define MC_HD inline
#endif

namespace mc {

constexpr int kTileRows = 16;
constexpr int kTileK = 128;
constexpr int kBlockRows = 128;   // rows of a supertile
constexpr int kTilesPerBlock = 8;
constexpr uint32_t kMagic = 0x4B50434Du;  // "MCPK"
constexpr uint32_t kFormatVersion = 3;
constexpr int kMaxE = 16;
constexpr int kHeaderBytes = 4096;

struct PackHeader {
    uint32_t magic;
    uint32_t version;
    int32_t E, H, F, group;
    int32_t reserved0, reserved1;
    int8_t bits[64];
    uint64_t mat_off[kMaxE][3];  // byte offset of each (expert, matrix) from the buffer start
    uint64_t total_bytes;
};
static_assert(sizeof(PackHeader) <= kHeaderBytes, "header");

MC_HD int tile_code_bytes(int bits) { return 256 * bits; }
MC_HD int tile_meta_bytes(int group) { return 64 * (kTileK / group); }
MC_HD int tile_bytes(int bits, int group) { return tile_code_bytes(bits) + tile_meta_bytes(group); }
MC_HD int supertile_bytes(int bits, int group) { return kTilesPerBlock * tile_bytes(bits, group); }
MC_HD uint64_t mat_bytes(int rows, int cols, int bits, int group)
{
    return (uint64_t)(rows / kTileRows) * (uint64_t)(cols / kTileK) * (uint64_t)tile_bytes(bits, group);
}
// Byte offset of supertile (128-row block rb, column step kt) of matrix m
// (0 = W1, 1 = W3: offsets inside the shared W1/W3 region; 2 = W2: inside the
// W2 region).  KT = column steps of the matrix, nrb = its 128-row blocks.
MC_HD uint64_t supertile_off(int m, int rb, int kt, int KT, int nrb, int STB)
{
    if (m < 2) return (((uint64_t)rb * KT + kt) * 2 + m) * (uint64_t)STB;
    const int pr = rb >> 1, pw = (2 * pr + 1 < nrb) ? 2 : 1;
    return ((uint64_t)pr * KT * 2 + (uint64_t)kt * pw + (rb & 1)) * (uint64_t)STB;
}
// supertiles per column step of W2 row-block pair pr
MC_HD int w2_pair_width(int pr, int nrb) { return (2 * pr + 1 < nrb) ? 2 : 1; }
// byte offset of tile (16-row block rb16, column step kt) of matrix m
MC_HD uint64_t tile_off(int m, int rb16, int kt, int KT, int nrb, int bits, int group)
{
    const int TB = tile_bytes(bits, group);
    return supertile_off(m, rb16 >> 3, kt, KT, nrb, kTilesPerBlock * TB) + (uint64_t)(rb16 & 7) * TB;
}

// row (0..15) and first column (0..127) of pair j of lane `lane` in a tile
MC_HD void pair_pos(int lane, int j, int &row, int &col)
{
    int g8 = lane >> 2, t = lane & 3, s = j >> 2, rho = j & 3;
    row = g8 + 8 * (rho & 1);
    col = 64 * (s >> 2) + 16 * t + 4 * (s & 3) + 2 * (rho >> 1);
}

// Inverse for the offset tables: pair index j of column `col` (0..127) for the
// rows of half `half` (0: rows 0..7, 1: rows 8..15).
MC_HD int pair_of_col(int col, int half)
{
    int h64 = col >> 6, s4 = (col >> 2) & 3, u2 = (col >> 1) & 1;
    int s = 4 * h64 + s4;
    return 4 * s + 2 * u2 + half;
}

// field position inside its word -> offset value 2^E
MC_HD int off2_pos(int j) { int p = j & 7; return p < 5 ? p : p - 5; }
MC_HD int off1_pos(int j) { int p = j & 15; return p < 10 ? p : p - 10; }
MC_HD float off2(int j) { return (float)(1 << (10 - 2 * off2_pos(j))); }
MC_HD float off1(int j) { return (float)(1 << (10 - off1_pos(j))); }

// Per (vector, group) table of 8 floats used by the expert kernels:
//   [0] X = sum of the group's fp16 inputs
//   [1],[2] O1 for row halves 0/1  (1-bit plane offsets)
//   [3],[4] O2 for row halves 0/1  (2-bit plane offsets)
//   [5],[6] O3 = O2 + 4*O1          (3-bit: low plane + 4 x high plane)
//   [7] unused
constexpr int kTabFloats = 8;

}  // namespace mc
