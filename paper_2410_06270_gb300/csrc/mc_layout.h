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
//   b = 1: 2 words, word i holds pairs 16i..16i+15; pair position p = j%16 has
//       its low-column code at bit p and its high-column code at bit 16+p.
//   b = 2: 4 words, word i holds pairs 8i..8i+7; position p = j%8 at bits
//       [2p, 2p+1] (low column) and [16+2p, 17+2p] (high column).
//   b = 3: 6 words.  Word i holds pairs 5i..5i+4 (i < 6, j < 30); position
//       p = j%5 has its low-column code at bits [f, f+2], f = 1, 4, 7, 10, 13
//       for p = 0..4, and its high-column code at bits [16+f, 18+f].  The
//       remaining bits 0 and 16 of the six words hold pairs 30 and 31: bit c of
//       the low- (high-) column code of pair 30 + u is bit 0 (16) of word 3u + c.
// Code bytes of a tile, lane-major inside each part:
//   b = 1: [32 lanes x 8 B]    b = 2: [32 lanes x 16 B]
//   b = 3: [32 lanes x 16 B: words 0..3][32 lanes x 8 B: words 4, 5]
// Meta bytes of a tile: [group-in-tile][g8 = 0..7][s(r0), z(r0), s(r1), z(r1)] fp16.
// 16-bit (unquantised) experts, b = 16: the tile holds the fp16 weights themselves,
// lane-major, 128 bytes per lane = its 32 pairs in order j (pair j = the two
// columns above, as one half2): a k-step's four A-fragment registers are one
// 16-byte load.  No meta.
//
// Decoding without shifts per field: a field at mantissa bit f of an fp16 whose
// exponent field is set to 15 + E reads as 2^E + q * 2^(E + f - 10); choosing
// E = 10 - f makes it (2^E + q).  Fields above the mantissa (bits 10..15 of a
// half) are first shifted down by 10.  The constant 2^E ("offset") depends only
// on the field position, so sum_k (off_k + q_k) x_k - sum_k off_k x_k
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
constexpr uint32_t kFormatVersion = 4;
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
MC_HD int tile_bytes(int bits, int group) { return tile_code_bytes(bits) + (bits == 16 ? 0 : tile_meta_bytes(group)); }
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

// Where bit c of the code of pair j sits for a lane: word index and bit inside
// it; h = 0 for the pair's low column, 1 for its high column.
MC_HD void code_bit(int bits, int j, int h, int c, int &word, int &bit)
{
    if (bits == 1) {
        word = j >> 4;
        bit = (j & 15) + 16 * h;
    } else if (bits == 2) {
        word = j >> 3;
        bit = 2 * (j & 7) + c + 16 * h;
    } else if (j < 30) {
        word = j / 5;
        bit = 1 + 3 * (j % 5) + c + 16 * h;
    } else {
        word = 3 * (j - 30) + c;
        bit = 16 * h;
    }
}
// byte offset of code word w of lane `lane` inside a tile
MC_HD int code_word_off(int bits, int lane, int w)
{
    if (bits == 1) return 8 * lane + 4 * w;
    if (bits == 2) return 16 * lane + 4 * w;
    return w < 4 ? 16 * lane + 4 * w : 512 + 8 * lane + 4 * (w - 4);
}

// mantissa bit of the field of pair j after the decoder's shift -> offset 2^E
MC_HD int off2_pos(int j) { int p = j & 7; return p < 5 ? p : p - 5; }
MC_HD int off1_pos(int j) { int p = j & 15; return p < 10 ? p : p - 10; }
MC_HD int off3_bit(int j)
{
    if (j >= 30) return 0;
    const int f = 1 + 3 * (j % 5);
    return f < 10 ? f : f - 10;
}
MC_HD float off2(int j) { return (float)(1 << (10 - 2 * off2_pos(j))); }
MC_HD float off1(int j) { return (float)(1 << (10 - off1_pos(j))); }
MC_HD float off3(int j) { return (float)(1 << (10 - off3_bit(j))); }

// Per (vector, group) table of 8 floats used by the tensor-core expert kernels:
//   [0] X = sum of the group's fp16 inputs
//   [1] unused
//   [2],[3] O1 for row halves 0/1  (sum of 1-bit offsets times the inputs)
//   [4],[5] O2 for row halves 0/1  (2-bit offsets)
//   [6],[7] O3 for row halves 0/1  (3-bit offsets)
constexpr int kTabFloats = 8;

}  // namespace mc
