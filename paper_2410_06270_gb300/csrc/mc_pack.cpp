// mc_pack.cpp -- host side of the PMQ weight storage (Sec. 2.2, App. A.2):
// canonical per-weight codes + fp16 scale/zero  <->  the packed tile layout of
// mc_layout.h, plus shape validation and the thread-local error text.
#include <string.h>

#include <algorithm>
#include <string>
#include <thread>
#include <vector>

#include "mc_host.h"

namespace mc {

static thread_local std::string g_err;

int set_error(int code, const char *fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_err = buf;
    return code;
}

void clear_error() { g_err.clear(); }

int check_shape(const mc_shape *s)
{
    if (!s) return set_error(MC_ERR_INVALID_ARG, "shape is NULL");
    if (s->top_k != 2) return set_error(MC_ERR_UNSUPPORTED, "top_k=%d: only top-2 routing is supported", s->top_k);
    if (s->E < 2 || s->E > kMaxE) return set_error(MC_ERR_UNSUPPORTED, "E=%d: need 2 <= E <= %d", s->E, kMaxE);
    if (s->group != 64 && s->group != 128)
        return set_error(MC_ERR_INVALID_ARG, "group=%d: need 64 or 128", s->group);
    if (s->H <= 0 || s->H % kTileK || s->H > 16384)
        return set_error(MC_ERR_INVALID_ARG, "H=%d: need a positive multiple of 128, <= 16384", s->H);
    if (s->F <= 0 || s->F % kTileK || s->F > 65536)
        return set_error(MC_ERR_INVALID_ARG, "F=%d: need a positive multiple of 128, <= 65536", s->F);
    return MC_OK;
}

int check_bits(const mc_shape *s, const int8_t *bits)
{
    int rc = check_shape(s);
    if (rc) return rc;
    if (!bits) return set_error(MC_ERR_INVALID_ARG, "bits table is NULL");
    int n16 = 0;
    for (int e = 0; e < s->E; ++e) {
        if (bits[e] == 16) {
            ++n16;
            continue;
        }
        if (bits[e] < 1 || bits[e] > 3)
            return set_error(MC_ERR_UNSUPPORTED, "bits[%d]=%d: only 1, 2, 3 or 16 bits are supported", e, bits[e]);
    }
    if (n16 && n16 != s->E)
        return set_error(MC_ERR_UNSUPPORTED, "16-bit experts cannot be mixed with quantised ones");
    return MC_OK;
}

void layout_offsets(const mc_shape *s, const int8_t *bits, uint64_t off[kMaxE][3], uint64_t *total)
{
    uint64_t pos = kHeaderBytes;
    for (int e = 0; e < s->E; ++e) {
        // W1 and W3 share one interleaved region; W2 follows
        off[e][0] = off[e][1] = pos;
        pos += 2 * mat_bytes(s->F, s->H, bits[e], s->group);
        pos = (pos + 255) & ~(uint64_t)255;
        off[e][2] = pos;
        pos += mat_bytes(s->H, s->F, bits[e], s->group);
        pos = (pos + 255) & ~(uint64_t)255;
    }
    *total = pos;
}

// Pack one matrix [rows, cols] into its tile stream.  Returns false on a code
// that does not fit in `bits`.
static void pack_dense(int m, int rows, int cols, const uint16_t *w, uint8_t *dst, int rb_lo, int rb_hi)
{
    const int KT = cols / kTileK, nrb = rows / kBlockRows;
    for (int rb = rb_lo; rb < rb_hi; ++rb)
        for (int kt = 0; kt < KT; ++kt) {
            uint16_t *tile = (uint16_t *)(dst + tile_off(m, rb, kt, KT, nrb, 16, kTileK));
            const int R0 = rb * kTileRows, K0 = kt * kTileK;
            for (int lane = 0; lane < 32; ++lane)
                for (int j = 0; j < 32; ++j) {
                    int row, col;
                    pair_pos(lane, j, row, col);
                    const uint16_t *src = w + (size_t)(R0 + row) * cols + K0 + col;
                    tile[lane * 64 + 2 * j] = src[0];
                    tile[lane * 64 + 2 * j + 1] = src[1];
                }
        }
}

static void unpack_dense(int m, int rows, int cols, const uint8_t *src, uint16_t *w)
{
    const int KT = cols / kTileK, nrb = rows / kBlockRows;
    for (int rb = 0; rb < rows / kTileRows; ++rb)
        for (int kt = 0; kt < KT; ++kt) {
            const uint16_t *tile = (const uint16_t *)(src + tile_off(m, rb, kt, KT, nrb, 16, kTileK));
            const int R0 = rb * kTileRows, K0 = kt * kTileK;
            for (int lane = 0; lane < 32; ++lane)
                for (int j = 0; j < 32; ++j) {
                    int row, col;
                    pair_pos(lane, j, row, col);
                    uint16_t *d = w + (size_t)(R0 + row) * cols + K0 + col;
                    d[0] = tile[lane * 64 + 2 * j];
                    d[1] = tile[lane * 64 + 2 * j + 1];
                }
        }
}

static bool pack_matrix(int m, int rows, int cols, int bits, int group, const uint8_t *codes,
                        const uint16_t *scale, const uint16_t *zero, uint8_t *dst, int rb_lo, int rb_hi)
{
    if (bits == 16) {
        pack_dense(m, rows, cols, (const uint16_t *)codes, dst, rb_lo, rb_hi);
        return true;
    }
    const int KT = cols / kTileK, ng = cols / group, gpt = kTileK / group, nrb = rows / kBlockRows;
    const uint32_t lim = 1u << bits;
    for (int rb = rb_lo; rb < rb_hi; ++rb)
        for (int kt = 0; kt < KT; ++kt) {
            uint8_t *tile = dst + tile_off(m, rb, kt, KT, nrb, bits, group);
            const int R0 = rb * kTileRows, K0 = kt * kTileK;
            for (int lane = 0; lane < 32; ++lane) {
                uint32_t w[6] = {0, 0, 0, 0, 0, 0};
                for (int j = 0; j < 32; ++j) {
                    int row, col;
                    pair_pos(lane, j, row, col);
                    const uint8_t *src = codes + (size_t)(R0 + row) * cols + K0 + col;
                    for (int h = 0; h < 2; ++h) {
                        const uint32_t q = src[h];
                        if (q >= lim) return false;
                        for (int c = 0; c < bits; ++c) {
                            int wi, bi;
                            code_bit(bits, j, h, c, wi, bi);
                            w[wi] |= ((q >> c) & 1u) << bi;
                        }
                    }
                }
                for (int wi = 0; wi < 2 * bits; ++wi) memcpy(tile + code_word_off(bits, lane, wi), &w[wi], 4);
            }
            uint16_t *meta = (uint16_t *)(tile + tile_code_bytes(bits));
            for (int gi = 0; gi < gpt; ++gi) {
                int gcol = (K0 + gi * group) / group;
                for (int g8 = 0; g8 < 8; ++g8) {
                    uint16_t *m4 = meta + (gi * 8 + g8) * 4;
                    size_t i0 = (size_t)(R0 + g8) * ng + gcol, i1 = (size_t)(R0 + g8 + 8) * ng + gcol;
                    m4[0] = scale[i0];
                    m4[1] = zero[i0];
                    m4[2] = scale[i1];
                    m4[3] = zero[i1];
                }
            }
        }
    return true;
}

static void unpack_matrix(int m, int rows, int cols, int bits, int group, const uint8_t *src,
                          uint8_t *codes, uint16_t *scale, uint16_t *zero)
{
    if (bits == 16) {
        unpack_dense(m, rows, cols, src, (uint16_t *)codes);
        return;
    }
    const int KT = cols / kTileK, ng = cols / group, gpt = kTileK / group, nrb = rows / kBlockRows;
    for (int rb = 0; rb < rows / kTileRows; ++rb)
        for (int kt = 0; kt < KT; ++kt) {
            const uint8_t *tile = src + tile_off(m, rb, kt, KT, nrb, bits, group);
            const int R0 = rb * kTileRows, K0 = kt * kTileK;
            for (int lane = 0; lane < 32; ++lane) {
                uint32_t w[6] = {0, 0, 0, 0, 0, 0};
                for (int wi = 0; wi < 2 * bits; ++wi) memcpy(&w[wi], tile + code_word_off(bits, lane, wi), 4);
                for (int j = 0; j < 32; ++j) {
                    int row, col;
                    pair_pos(lane, j, row, col);
                    uint8_t *d = codes + (size_t)(R0 + row) * cols + K0 + col;
                    for (int h = 0; h < 2; ++h) {
                        uint32_t q = 0;
                        for (int c = 0; c < bits; ++c) {
                            int wi, bi;
                            code_bit(bits, j, h, c, wi, bi);
                            q |= ((w[wi] >> bi) & 1u) << c;
                        }
                        d[h] = (uint8_t)q;
                    }
                }
            }
            const uint16_t *meta = (const uint16_t *)(tile + tile_code_bytes(bits));
            for (int gi = 0; gi < gpt; ++gi) {
                int gcol = (K0 + gi * group) / group;
                for (int g8 = 0; g8 < 8; ++g8) {
                    const uint16_t *m4 = meta + (gi * 8 + g8) * 4;
                    size_t i0 = (size_t)(R0 + g8) * ng + gcol, i1 = (size_t)(R0 + g8 + 8) * ng + gcol;
                    if (scale) { scale[i0] = m4[0]; scale[i1] = m4[2]; }
                    if (zero) { zero[i0] = m4[1]; zero[i1] = m4[3]; }
                }
            }
        }
}

}  // namespace mc

using namespace mc;

extern "C" {

size_t mc_packed_size(const mc_shape *shape, const int8_t *bits_host)
{
    if (check_bits(shape, bits_host)) return 0;
    uint64_t off[kMaxE][3], total;
    layout_offsets(shape, bits_host, off, &total);
    return (size_t)total;
}

int mc_pack_experts_host(const mc_shape *shape, const int8_t *bits_host,
                         const uint8_t *const *codes_host, const uint16_t *const *scale_host,
                         const uint16_t *const *zero_host, void *packed_host, size_t packed_bytes)
{
    clear_error();
    int rc = check_bits(shape, bits_host);
    if (rc) return rc;
    if (!codes_host || !scale_host || !zero_host || !packed_host)
        return set_error(MC_ERR_INVALID_ARG, "NULL array argument");
    uint64_t off[kMaxE][3], total;
    layout_offsets(shape, bits_host, off, &total);
    if (packed_bytes < total)
        return set_error(MC_ERR_INVALID_ARG, "packed buffer has %zu bytes, needs %llu", packed_bytes,
                         (unsigned long long)total);
    for (int i = 0; i < 3 * shape->E; ++i)
        if (!codes_host[i] || (bits_host[i / 3] != 16 && (!scale_host[i] || !zero_host[i])))
            return set_error(MC_ERR_INVALID_ARG, "NULL array for expert %d matrix %d", i / 3, i % 3);
    uint8_t *base = (uint8_t *)packed_host;
    memset(base, 0, kHeaderBytes);
    PackHeader *hd = (PackHeader *)base;
    hd->magic = kMagic;
    hd->version = kFormatVersion;
    hd->E = shape->E;
    hd->H = shape->H;
    hd->F = shape->F;
    hd->group = shape->group;
    for (int e = 0; e < shape->E; ++e) {
        hd->bits[e] = bits_host[e];
        for (int m = 0; m < 3; ++m) hd->mat_off[e][m] = off[e][m];
    }
    hd->total_bytes = total;

    // one work item per (expert, matrix, 128-row block), spread over host threads
    struct Item { int e, m, rb_lo, rb_hi; };
    std::vector<Item> items;
    for (int e = 0; e < shape->E; ++e)
        for (int m = 0; m < 3; ++m) {
            int rows = m < 2 ? shape->F : shape->H;
            for (int r = 0; r < rows / kTileRows; r += 8) items.push_back({e, m, r, std::min(r + 8, rows / kTileRows)});
        }
    unsigned nth = std::max(1u, std::min(32u, std::thread::hardware_concurrency()));
    std::vector<int> bad(nth, -1);
    auto work = [&](unsigned id) {
        for (size_t i = id; i < items.size(); i += nth) {
            const Item &it = items[i];
            int rows = it.m < 2 ? shape->F : shape->H, cols = it.m < 2 ? shape->H : shape->F;
            int k = 3 * it.e + it.m;
            if (!pack_matrix(it.m, rows, cols, bits_host[it.e], shape->group, codes_host[k], scale_host[k],
                             zero_host[k], base + off[it.e][it.m], it.rb_lo, it.rb_hi)) {
                bad[id] = k;
                return;
            }
        }
    };
    std::vector<std::thread> th;
    for (unsigned i = 1; i < nth; ++i) th.emplace_back(work, i);
    work(0);
    for (auto &t : th) t.join();
    for (unsigned i = 0; i < nth; ++i)
        if (bad[i] >= 0)
            return set_error(MC_ERR_INVALID_ARG, "expert %d matrix %d has a code >= 2^%d", bad[i] / 3, bad[i] % 3,
                             bits_host[bad[i] / 3]);
    return MC_OK;
}

int mc_unpack_experts_host(const void *packed_host, size_t packed_bytes, int expert, int mat,
                           uint8_t *codes_host, uint16_t *scale_host, uint16_t *zero_host)
{
    clear_error();
    if (!packed_host || !codes_host) return set_error(MC_ERR_INVALID_ARG, "NULL argument");
    if (packed_bytes < (size_t)kHeaderBytes) return set_error(MC_ERR_BAD_PACK, "buffer shorter than the header");
    const PackHeader *hd = (const PackHeader *)packed_host;
    if (hd->magic != kMagic || hd->version != kFormatVersion)
        return set_error(MC_ERR_BAD_PACK, "bad magic/version (%08x/%u)", hd->magic, hd->version);
    mc_shape s = {hd->E, hd->H, hd->F, hd->group, 2};
    int rc = check_bits(&s, hd->bits);
    if (rc) return set_error(MC_ERR_BAD_PACK, "header: %s", mc_last_error());
    if (hd->total_bytes > packed_bytes) return set_error(MC_ERR_BAD_PACK, "buffer shorter than header total");
    if (expert < 0 || expert >= hd->E || mat < 0 || mat > 2)
        return set_error(MC_ERR_INVALID_ARG, "expert %d / matrix %d out of range", expert, mat);
    int rows = mat < 2 ? hd->F : hd->H, cols = mat < 2 ? hd->H : hd->F;
    unpack_matrix(mat, rows, cols, hd->bits[expert], hd->group,
                  (const uint8_t *)packed_host + hd->mat_off[expert][mat], codes_host, scale_host, zero_host);
    return MC_OK;
}

const char *mc_last_error(void) { return g_err.c_str(); }

int mc_version(void) { return 10000; }
int mc_pack_format_version(void) { return (int)kFormatVersion; }

}  // extern "C"
