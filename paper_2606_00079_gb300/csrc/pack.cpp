// Host packer / unpacker of the bucketed BitsMoE layer image (no CUDA here).
//
// Stored unit format (reading of the paper's quantiser, Eq.
// app_scalar_quantization_uk with one fp16 scale and zero per group of 128 in
// the experiments): code q in [0, 2^b), p_hat = scale * (q - zero); b = 16 units
// are fp16 values; 0-bit units are evicted (Eq. app_zero_bit_vector) and are
// not stored at all.  The layout itself is described in format.h.
#include <algorithm>
#include <atomic>
#include <cstdlib>
#include <cstring>
#include <new>
#include <thread>
#include <vector>

#include "internal.h"

namespace bmoe {
namespace {

struct Dims {
  int D, E, I, n, group, D_pad, n_pad, I_pad, NRB, NG;
};

struct Plane {   // one bit-plane chunk of a tile
  int pb;        // bits per code in this plane
  int pshift;    // position of the plane inside the code
  int base;      // RL: first unit of the tile in this chunk; UL: first row of the row block
};

// RL (gate/up) chunk -> plane
Plane rl_plane(int b, int chunk) {
  if (b == 3) return chunk < 2 ? Plane{2, 0, 16 * chunk} : Plane{1, 2, 0};
  if (b == 6) return chunk < 2 ? Plane{4, 0, 8 * chunk} : Plane{2, 4, 0};
  return Plane{b, 0, 0};
}
// UL (down) chunk -> plane
Plane ul_plane(int b, int chunk) {
  if (b == 3) return chunk < 2 ? Plane{2, 0, 64 * chunk} : Plane{1, 2, 0};
  if (b == 6) return chunk < 4 ? Plane{4, 0, 32 * chunk} : Plane{2, 4, 64 * (chunk - 4)};
  return Plane{b, 0, chunk * (kRows / b)};
}

// Enumerate every (word, bit position, plane, slot, row) of one bucket's stream.
// f(word_index_in_stream, bitpos, plane_bits, plane_shift, slot, row).
template <class F>
void visit_rl(int b, int ntiles, int NRB, uint64_t rb_stride_words, uint64_t bucket_word_off, F&& f) {
  const int U = rl_units(b), C = rl_chunks(b);
  for (int rb = 0; rb < NRB; ++rb)
    for (int tile = 0; tile < ntiles; ++tile)
      for (int c = 0; c < C; ++c)
        for (int lane = 0; lane < 32; ++lane)
          for (int w = 0; w < 4; ++w) {
            const uint64_t word = rb * rb_stride_words + bucket_word_off +
                                  ((uint64_t)(tile * C + c) * 32 + lane) * 4 + w;
            const int row = rb * kRows + 4 * lane + w;
            if (b == 16) {
              f(word, 0, 16, 0, tile * U + 2 * c, row);
              f(word, 16, 16, 0, tile * U + 2 * c + 1, row);
              continue;
            }
            const Plane p = rl_plane(b, c);
            const int nu = 32 / p.pb;
            for (int u = 0; u < nu; ++u)
              f(word, 8 * (u % 4) + p.pb * (u / 4), p.pb, p.pshift, tile * U + p.base + u, row);
          }
}

template <class F>
void visit_ul(int b, int ntiles, int NRB, uint64_t bucket_word_off, F&& f) {
  const int C = ul_chunks(b);
  for (int tile = 0; tile < ntiles; ++tile)
    for (int rb = 0; rb < NRB; ++rb)
      for (int c = 0; c < C; ++c)
        for (int lane = 0; lane < 32; ++lane)
          for (int w = 0; w < 4; ++w) {
            const uint64_t word = bucket_word_off +
                                  (((uint64_t)tile * NRB + rb) * C + c) * 128 + lane * 4 + w;
            const int slot = tile * 32 + lane;
            if (b == 16) {
              const int r0 = rb * kRows + 8 * c + 2 * w;
              f(word, 0, 16, 0, slot, r0);
              f(word, 16, 16, 0, slot, r0 + 1);
              continue;
            }
            const Plane p = ul_plane(b, c);
            const int rpw = 32 / p.pb;
            for (int r = 0; r < rpw; ++r)
              f(word, 8 * (r % 4) + p.pb * (r / 4), p.pb, p.pshift, slot,
                rb * kRows + p.base + w * rpw + r);
          }
}

int check_dims(const bitsmoe_layer_host* s, Dims& d) {
  if (!s) return BITSMOE_ERR_INVALID_ARG;
  if (s->D < 1 || s->E < 1 || s->E > 1024 || s->I < 1 || s->n < 1 || s->n > 65535)
    return BITSMOE_ERR_SHAPE;
  if (!group_ok(s->group) || s->I % s->group) return BITSMOE_ERR_SHAPE;
  if (s->D > (1 << 20) || s->I > (1 << 22)) return BITSMOE_ERR_SHAPE;
  for (int h = 0; h < 3; ++h)
    if (!s->basis[h]) return BITSMOE_ERR_INVALID_ARG;
  if (!s->bits || !s->alpha || !s->codes || !s->scale || !s->zero) return BITSMOE_ERR_INVALID_ARG;
  d.D = s->D; d.E = s->E; d.I = s->I; d.n = s->n; d.group = s->group;
  d.D_pad = (int)align_up(d.D, 8);
  d.n_pad = (int)align_up(d.n, 8);
  d.I_pad = (int)align_up(d.I, std::max(kRows, d.group));
  d.NRB = d.I_pad / kRows;
  d.NG = d.I_pad / d.group;
  return BITSMOE_OK;
}

struct Plan {
  int h, e;
  std::vector<int> units[kNumBk];   // unit indices per bucket, increasing j
};

template <class F>
void parallel_for(int count, F&& f) {
  unsigned nt = std::thread::hardware_concurrency();
  nt = std::max(1u, std::min(nt, 32u));
  if (count < 2 || nt == 1) {
    for (int i = 0; i < count; ++i) f(i);
    return;
  }
  std::vector<std::thread> th;
  std::atomic_int next{0};
  for (unsigned t = 0; t < nt; ++t)
    th.emplace_back([&] {
      for (int i = next++; i < count; i = next++) f(i);
    });
  for (auto& t : th) t.join();
}

}  // namespace

int build_image(const bitsmoe_layer_host* src, std::vector<uint8_t>& img) {
  Dims d;
  int rc = check_dims(src, d);
  if (rc) return rc;
  const int E = d.E, n = d.n, I = d.I;
  const int ngroups_real = I / d.group;

  // 1. bucket the units of every (h, e)
  std::vector<Plan> plans(3 * (size_t)E);
  for (int h = 0; h < 3; ++h)
    for (int e = 0; e < E; ++e) {
      Plan& p = plans[h * E + e];
      p.h = h; p.e = e;
      const uint8_t* bits = src->bits + ((size_t)h * E + e) * n;
      for (int j = 0; j < n; ++j) {
        const int b = bits[j];
        if (!bits_ok(b)) return BITSMOE_ERR_UNSUPPORTED_BITS;
        if (b) p.units[bk_of_bits(b)].push_back(j);
      }
    }

  // codes of quantised units must lie in [0, 2^b)
  {
    std::atomic_int bad{0};
    parallel_for(3 * E, [&](int pi) {
      const uint8_t* bits = src->bits + (size_t)pi * n;
      for (int j = 0; j < n && !bad.load(std::memory_order_relaxed); ++j) {
        const int b = bits[j];
        if (b == 0 || b == 16) continue;
        const uint16_t* q = src->codes + ((size_t)pi * n + j) * I;
        uint32_t acc = 0;
        for (int i = 0; i < I; ++i) acc |= q[i];
        if (acc >> b) bad = 1;
      }
    });
    if (bad) return BITSMOE_ERR_INVALID_ARG;
  }

  // 2. descriptors and sizes
  std::vector<ExpertDesc> desc(3 * (size_t)E);
  uint64_t max_rb_stride = 0;
  int ul_max_tiles = 0;
  for (size_t pi = 0; pi < plans.size(); ++pi) {
    const Plan& p = plans[pi];
    ExpertDesc& x = desc[pi];
    std::memset(&x, 0, sizeof(x));
    const bool rl = p.h < 2;
    int slot = 0, tile = 0;
    uint64_t off = 0;
    for (int k = 0; k < kNumBk; ++k) {
      const int cnt = (int)p.units[k].size();
      if (!cnt) continue;
      const int b = bk_bits(k);
      BucketDesc& bd = x.bk[x.nbk++];
      bd.bits = b;
      bd.count = cnt;
      const int per_tile = rl ? rl_units(b) : 32;
      bd.ntiles = (cnt + per_tile - 1) / per_tile;
      bd.nslots = bd.ntiles * per_tile;
      bd.slot0 = slot;
      bd.tile0 = tile;
      bd.code_off = off;
      off += rl ? (uint64_t)bd.ntiles * rl_chunks(b) * kChunkBytes
                : (uint64_t)bd.ntiles * d.NRB * ul_chunks(b) * kChunkBytes;
      slot += bd.nslots;
      tile += bd.ntiles;
      x.nunits += cnt;
      // algorithmic bytes: codes, fp16 scale+zero per group (quantised units), fp32 alpha
      x.moved += ((uint64_t)cnt * I * b) / 8 + (b < 16 ? (uint64_t)cnt * ngroups_real * 4 : 0) +
                 (uint64_t)cnt * 4;
    }
    x.nslots = slot;
    x.ntiles = tile;
    x.rb_stride = off;
    if (rl) max_rb_stride = std::max(max_rb_stride, off);
    else ul_max_tiles = std::max(ul_max_tiles, tile);
  }

  // K2 segments: ~4 KB of codes per segment and row block
  int nseg = (int)std::min<uint64_t>(64, std::max<uint64_t>(1, (max_rb_stride + 4095) / 4096));
  std::vector<int32_t> seg(2 * (size_t)E * (nseg + 1), 0);
  int seg_max_slots = 0;
  for (int h = 0; h < 2; ++h)
    for (int e = 0; e < E; ++e) {
      const ExpertDesc& x = desc[h * E + e];
      int32_t* sg = &seg[((size_t)h * E + e) * (nseg + 1)];
      // flat tile sizes
      std::vector<uint64_t> cum(1, 0);
      std::vector<int> units_of_tile;
      for (int k = 0; k < x.nbk; ++k)
        for (int t = 0; t < x.bk[k].ntiles; ++t) {
          cum.push_back(cum.back() + (uint64_t)rl_chunks(x.bk[k].bits) * kChunkBytes);
          units_of_tile.push_back(rl_units(x.bk[k].bits));
        }
      const uint64_t total = cum.back();
      int t = 0;
      sg[0] = 0;
      for (int s = 1; s < nseg; ++s) {
        const uint64_t target = total * s / nseg;
        while (t < x.ntiles && cum[t] < target) ++t;
        sg[s] = t;
      }
      sg[nseg] = x.ntiles;
      for (int s = 0; s < nseg; ++s) {
        int sl = 0;
        for (int q = sg[s]; q < sg[s + 1]; ++q) sl += units_of_tile[q];
        seg_max_slots = std::max(seg_max_slots, sl);
      }
    }

  // 3. image offsets
  ImageHeader hd;
  std::memset(&hd, 0, sizeof(hd));
  hd.magic = kMagic; hd.version = kVersion;
  hd.D = d.D; hd.E = E; hd.I = I; hd.n = n; hd.group = d.group;
  hd.D_pad = d.D_pad; hd.n_pad = d.n_pad; hd.I_pad = d.I_pad; hd.NRB = d.NRB; hd.NG = d.NG;
  hd.nseg = nseg; hd.seg_max_slots = seg_max_slots; hd.ul_max_tiles = ul_max_tiles;
  uint64_t off = align_up(sizeof(ImageHeader), 256);
  hd.off_desc = off;      off = align_up(off + desc.size() * sizeof(ExpertDesc), 256);
  hd.off_seg = off;       off = align_up(off + seg.size() * sizeof(int32_t), 256);
  hd.off_items = off;     off = align_up(off + 2ull * E * nseg * sizeof(ItemRec), 256);
  hd.off_basis_in = off;  off = align_up(off + 2ull * n * d.D_pad * 2, 256);
  hd.off_basis_out = off; off = align_up(off + (uint64_t)d.D * d.n_pad * 2, 256);
  for (size_t pi = 0; pi < desc.size(); ++pi) {
    ExpertDesc& x = desc[pi];
    x.begin = off;
    x.unit_off = off;  off = align_up(off + (uint64_t)x.nslots * 4, 16);
    x.alpha_off = off; off = align_up(off + (uint64_t)x.nslots * 4, 16);
    x.sz_off = off;    off = align_up(off + (uint64_t)d.NG * x.nslots * 4, 16);
    for (int k = 0; k < x.nbk; ++k) x.bk[k].sz_off = x.sz_off + (uint64_t)x.bk[k].slot0 * 4;
    hd.meta_bytes += off - x.begin;
    off = align_up(off, 256);
    x.code_base = off;
    const uint64_t stream = pi < 2 * (size_t)E ? x.rb_stride * d.NRB : x.rb_stride;
    off = align_up(off + stream, 256);
    hd.codes_bytes += stream;
    x.end = off;
  }
  hd.total_bytes = off;

  try {
    img.assign(off, 0);
  } catch (const std::bad_alloc&) {
    return BITSMOE_ERR_OOM;
  }
  uint8_t* base = img.data();
  std::memcpy(base, &hd, sizeof(hd));
  std::memcpy(base + hd.off_desc, desc.data(), desc.size() * sizeof(ExpertDesc));
  std::memcpy(base + hd.off_seg, seg.data(), seg.size() * sizeof(int32_t));
  // gate/up item table
  {
    ItemRec* items = reinterpret_cast<ItemRec*>(base + hd.off_items);
    for (int pi = 0; pi < 2 * E; ++pi) {
      const ExpertDesc& x = desc[pi];
      const int32_t* sg = &seg[(size_t)pi * (nseg + 1)];
      for (int q = 0; q < nseg; ++q) {
        ItemRec& it = items[(size_t)pi * nseg + q];
        std::memset(&it, 0, sizeof(it));
        const int t0 = sg[q], t1 = sg[q + 1];
        for (int k = 0; k < x.nbk; ++k) {
          const BucketDesc& bd = x.bk[k];
          const int lo = std::max(t0, bd.tile0) - bd.tile0, hi = std::min(t1, bd.tile0 + bd.ntiles) - bd.tile0;
          if (lo >= hi) continue;
          if (it.nr == 0) {
            it.bk0 = (uint8_t)k;
            it.byte0 = (uint32_t)(bd.code_off + (uint64_t)lo * rl_chunks(bd.bits) * kChunkBytes);
            it.slot0 = (uint32_t)(bd.slot0 + lo * rl_units(bd.bits));
          }
          it.bits[it.nr] = (uint8_t)bd.bits;
          it.ntl[it.nr] = (uint16_t)(hi - lo);
          it.bytes += (uint32_t)((hi - lo) * rl_chunks(bd.bits) * kChunkBytes);
          it.nslot = (uint16_t)(it.nslot + (hi - lo) * rl_units(bd.bits));
          ++it.nr;
        }
      }
    }
  }

  // 4. bases
  uint16_t* bin = reinterpret_cast<uint16_t*>(base + hd.off_basis_in);
  for (int h = 0; h < 2; ++h)
    for (int dd = 0; dd < d.D; ++dd) {
      const uint16_t* row = src->basis[h] + (size_t)dd * n;
      for (int j = 0; j < n; ++j) bin[((size_t)h * n + j) * d.D_pad + dd] = row[j];
    }
  uint16_t* bout = reinterpret_cast<uint16_t*>(base + hd.off_basis_out);
  for (int dd = 0; dd < d.D; ++dd)
    std::memcpy(bout + (size_t)dd * d.n_pad, src->basis[2] + (size_t)dd * n, (size_t)n * 2);

  // 5. per (h, e) metadata and code streams
  parallel_for((int)plans.size(), [&](int pi) {
    const Plan& p = plans[pi];
    const ExpertDesc& x = desc[pi];
    const size_t he = (size_t)p.h * E + p.e;
    int32_t* unit = reinterpret_cast<int32_t*>(base + x.unit_off);
    float* alpha = reinterpret_cast<float*>(base + x.alpha_off);
    uint32_t* words = reinterpret_cast<uint32_t*>(base + x.code_base);
    int kk = 0;
    for (int k = 0; k < kNumBk; ++k) {
      if (p.units[k].empty()) continue;
      const BucketDesc& bd = x.bk[kk++];
      const std::vector<int>& us = p.units[k];
      for (int s = 0; s < bd.nslots; ++s) {
        unit[bd.slot0 + s] = s < bd.count ? us[s] : 0;
        alpha[bd.slot0 + s] = s < bd.count ? src->alpha[he * n + us[s]] : 0.0f;
      }
      if (bd.bits < 16) {
        uint32_t* sz = reinterpret_cast<uint32_t*>(base + bd.sz_off);
        for (int g = 0; g < ngroups_real; ++g)
          for (int s = 0; s < bd.count; ++s) {
            const size_t q = (he * n + us[s]) * ngroups_real + g;
            sz[(size_t)g * x.nslots + s] = (uint32_t)src->scale[q] | ((uint32_t)src->zero[q] << 16);
          }
      }
      auto put = [&](uint64_t word, int bitpos, int pb, int pshift, int slot, int row) {
        if (slot >= bd.count || row >= I) return;
        const uint32_t q = src->codes[(he * n + us[slot]) * I + row];
        const uint32_t mask = pb == 16 ? 0xFFFFu : ((1u << pb) - 1);
        words[word] |= ((q >> pshift) & mask) << bitpos;
      };
      if (p.h < 2)
        visit_rl(bd.bits, bd.ntiles, d.NRB, x.rb_stride / 4, bd.code_off / 4, put);
      else
        visit_ul(bd.bits, bd.ntiles, d.NRB, bd.code_off / 4, put);
    }
  });
  return BITSMOE_OK;
}

int validate_image(const uint8_t* img, size_t bytes) {
  if (!img || bytes < sizeof(ImageHeader)) return BITSMOE_ERR_BLOB;
  const ImageHeader* hd = header_of(img);
  if (hd->magic != kMagic || hd->version != kVersion || hd->total_bytes != bytes) return BITSMOE_ERR_BLOB;
  const int E = hd->E, n = hd->n, I = hd->I;
  if (hd->D < 1 || E < 1 || E > 1024 || I < 1 || n < 1 || n > 65535 || !group_ok(hd->group) ||
      I % hd->group)
    return BITSMOE_ERR_BLOB;
  if (hd->D_pad != (int)align_up(hd->D, 8) || hd->n_pad != (int)align_up(n, 8) ||
      hd->I_pad != (int)align_up(I, std::max(kRows, hd->group)) || hd->NRB != hd->I_pad / kRows ||
      hd->NG != hd->I_pad / hd->group || hd->nseg < 1 || hd->nseg > 64)
    return BITSMOE_ERR_BLOB;
  auto in = [&](uint64_t off, uint64_t len) { return off <= bytes && len <= bytes - off; };
  if (!in(hd->off_desc, 3ull * E * sizeof(ExpertDesc)) ||
      !in(hd->off_seg, 2ull * E * (hd->nseg + 1) * 4) ||
      !in(hd->off_items, 2ull * E * hd->nseg * sizeof(ItemRec)) || hd->off_items % 16 ||
      !in(hd->off_basis_in, 2ull * n * hd->D_pad * 2) ||
      !in(hd->off_basis_out, (uint64_t)hd->D * hd->n_pad * 2))
    return BITSMOE_ERR_BLOB;
  if (hd->off_desc % 16 || hd->off_basis_in % 16 || hd->off_basis_out % 16) return BITSMOE_ERR_BLOB;
  const ExpertDesc* desc = desc_of(img);
  const int32_t* seg = reinterpret_cast<const int32_t*>(img + hd->off_seg);
  int ul_max_tiles = 0;
  for (int pi = 0; pi < 3 * E; ++pi) {
    const ExpertDesc& x = desc[pi];
    const bool rl = pi < 2 * E;
    if (x.nbk < 0 || x.nbk > kNumBk) return BITSMOE_ERR_BLOB;
    if (!in(x.unit_off, (uint64_t)x.nslots * 4) || !in(x.alpha_off, (uint64_t)x.nslots * 4) ||
        !in(x.sz_off, (uint64_t)hd->NG * x.nslots * 4) || x.unit_off % 16 || x.alpha_off % 16 ||
        x.sz_off % 16 || x.code_base % 16 || x.nslots % 4)
      return BITSMOE_ERR_BLOB;
    const uint64_t stream = rl ? x.rb_stride * hd->NRB : x.rb_stride;
    if (!in(x.code_base, stream)) return BITSMOE_ERR_BLOB;
    int slot = 0, tile = 0, units = 0, prev_k = -1;
    uint64_t off = 0;
    for (int k = 0; k < x.nbk; ++k) {
      const BucketDesc& bd = x.bk[k];
      const int bk = bk_of_bits(bd.bits);
      if (bk <= prev_k) return BITSMOE_ERR_BLOB;
      prev_k = bk;
      const int per_tile = rl ? rl_units(bd.bits) : 32;
      if (bd.count < 1 || bd.ntiles != (bd.count + per_tile - 1) / per_tile ||
          bd.nslots != bd.ntiles * per_tile || bd.slot0 != slot || bd.tile0 != tile ||
          bd.code_off != off)
        return BITSMOE_ERR_BLOB;
      if (bd.sz_off != x.sz_off + (uint64_t)bd.slot0 * 4) return BITSMOE_ERR_BLOB;
      off += rl ? (uint64_t)bd.ntiles * rl_chunks(bd.bits) * kChunkBytes
                : (uint64_t)bd.ntiles * hd->NRB * ul_chunks(bd.bits) * kChunkBytes;
      slot += bd.nslots;
      tile += bd.ntiles;
      units += bd.count;
    }
    if (slot != x.nslots || tile != x.ntiles || units != x.nunits || off != x.rb_stride)
      return BITSMOE_ERR_BLOB;
    const int32_t* unit = reinterpret_cast<const int32_t*>(img + x.unit_off);
    for (int s = 0; s < x.nslots; ++s)
      if (unit[s] < 0 || unit[s] >= n) return BITSMOE_ERR_BLOB;
    if (rl) {
      const ItemRec* items = reinterpret_cast<const ItemRec*>(img + hd->off_items) + (size_t)pi * hd->nseg;
      const int32_t* sg = seg + (size_t)pi * (hd->nseg + 1);
      for (int q = 0; q < hd->nseg; ++q) {   // item records must match the segment table
        const ItemRec& it = items[q];
        int nr = 0, slots = 0;
        uint64_t bytes = 0;
        for (int k = 0; k < x.nbk; ++k) {
          const BucketDesc& bd = x.bk[k];
          const int lo = std::max(sg[q], bd.tile0) - bd.tile0, hi = std::min(sg[q + 1], bd.tile0 + bd.ntiles) - bd.tile0;
          if (lo >= hi) continue;
          if (nr == 0 && (it.bk0 != k || it.byte0 != bd.code_off + (uint64_t)lo * rl_chunks(bd.bits) * kChunkBytes ||
                          it.slot0 != (uint32_t)(bd.slot0 + lo * rl_units(bd.bits))))
            return BITSMOE_ERR_BLOB;
          if (nr >= kNumBk || it.bits[nr] != bd.bits || it.ntl[nr] != hi - lo) return BITSMOE_ERR_BLOB;
          bytes += (uint64_t)(hi - lo) * rl_chunks(bd.bits) * kChunkBytes;
          slots += (hi - lo) * rl_units(bd.bits);
          ++nr;
        }
        if (it.nr != nr || it.bytes != bytes || it.nslot != slots) return BITSMOE_ERR_BLOB;
      }
      if (sg[0] != 0 || sg[hd->nseg] != x.ntiles) return BITSMOE_ERR_BLOB;
      for (int s = 0; s < hd->nseg; ++s)
        if (sg[s + 1] < sg[s]) return BITSMOE_ERR_BLOB;
      for (int s = 0; s < hd->nseg; ++s) {
        int sl = 0;
        for (int k = 0; k < x.nbk; ++k) {
          const BucketDesc& bd = x.bk[k];
          const int lo = std::max(sg[s], bd.tile0), hi = std::min(sg[s + 1], bd.tile0 + bd.ntiles);
          if (hi > lo) sl += (hi - lo) * rl_units(bd.bits);
        }
        if (sl > hd->seg_max_slots) return BITSMOE_ERR_BLOB;
      }
    } else {
      ul_max_tiles = std::max(ul_max_tiles, x.ntiles);
    }
  }
  if (ul_max_tiles != hd->ul_max_tiles) return BITSMOE_ERR_BLOB;
  return BITSMOE_OK;
}

int unpack_image(const uint8_t* img, size_t bytes, bitsmoe_layer_host_out* dst) {
  int rc = validate_image(img, bytes);
  if (rc) return rc;
  const ImageHeader* hd = header_of(img);
  if (!dst || dst->D != hd->D || dst->E != hd->E || dst->I != hd->I || dst->n != hd->n ||
      dst->group != hd->group)
    return BITSMOE_ERR_SHAPE;
  for (int h = 0; h < 3; ++h)
    if (!dst->basis[h]) return BITSMOE_ERR_INVALID_ARG;
  if (!dst->bits || !dst->alpha || !dst->codes || !dst->scale || !dst->zero) return BITSMOE_ERR_INVALID_ARG;
  const int D = hd->D, E = hd->E, I = hd->I, n = hd->n, ng = I / hd->group;
  const uint16_t* bin = reinterpret_cast<const uint16_t*>(img + hd->off_basis_in);
  for (int h = 0; h < 2; ++h)
    for (int dd = 0; dd < D; ++dd)
      for (int j = 0; j < n; ++j)
        dst->basis[h][(size_t)dd * n + j] = bin[((size_t)h * n + j) * hd->D_pad + dd];
  const uint16_t* bout = reinterpret_cast<const uint16_t*>(img + hd->off_basis_out);
  for (int dd = 0; dd < D; ++dd)
    std::memcpy(dst->basis[2] + (size_t)dd * n, bout + (size_t)dd * hd->n_pad, (size_t)n * 2);
  std::memset(dst->bits, 0, 3ull * E * n);
  std::memset(dst->alpha, 0, 3ull * E * n * 4);
  std::memset(dst->codes, 0, 3ull * E * n * I * 2);
  std::memset(dst->scale, 0, 3ull * E * n * ng * 2);
  std::memset(dst->zero, 0, 3ull * E * n * ng * 2);
  const ExpertDesc* desc = desc_of(img);
  parallel_for(3 * E, [&](int pi) {
    const ExpertDesc& x = desc[pi];
    const size_t he = (size_t)pi;
    const int32_t* unit = reinterpret_cast<const int32_t*>(img + x.unit_off);
    const float* alpha = reinterpret_cast<const float*>(img + x.alpha_off);
    const uint32_t* words = reinterpret_cast<const uint32_t*>(img + x.code_base);
    for (int k = 0; k < x.nbk; ++k) {
      const BucketDesc& bd = x.bk[k];
      for (int s = 0; s < bd.count; ++s) {
        const int j = unit[bd.slot0 + s];
        dst->bits[he * n + j] = (uint8_t)bd.bits;
        dst->alpha[he * n + j] = alpha[bd.slot0 + s];
      }
      if (bd.bits < 16) {
        const uint32_t* sz = reinterpret_cast<const uint32_t*>(img + bd.sz_off);
        for (int g = 0; g < ng; ++g)
          for (int s = 0; s < bd.count; ++s) {
            const int j = unit[bd.slot0 + s];
            const uint32_t v = sz[(size_t)g * x.nslots + s];
            dst->scale[(he * n + j) * ng + g] = (uint16_t)(v & 0xFFFF);
            dst->zero[(he * n + j) * ng + g] = (uint16_t)(v >> 16);
          }
      }
      auto get = [&](uint64_t word, int bitpos, int pb, int pshift, int slot, int row) {
        if (slot >= bd.count || row >= I) return;
        const int j = unit[bd.slot0 + slot];
        const uint32_t mask = pb == 16 ? 0xFFFFu : ((1u << pb) - 1);
        dst->codes[(he * n + j) * I + row] |= (uint16_t)(((words[word] >> bitpos) & mask) << pshift);
      };
      if (pi < 2 * E)
        visit_rl(bd.bits, bd.ntiles, hd->NRB, x.rb_stride / 4, bd.code_off / 4, get);
      else
        visit_ul(bd.bits, bd.ntiles, hd->NRB, bd.code_off / 4, get);
    }
  });
  return BITSMOE_OK;
}

}  // namespace bmoe

extern "C" {

int bitsmoe_pack_to_host(const bitsmoe_layer_host* src, void** blob, size_t* bytes) {
  if (!src || !blob || !bytes) return BITSMOE_ERR_INVALID_ARG;
  *blob = nullptr;
  *bytes = 0;
  std::vector<uint8_t> img;
  int rc = bmoe::build_image(src, img);
  if (rc) return rc;
  void* p = std::malloc(img.size());
  if (!p) return BITSMOE_ERR_OOM;
  std::memcpy(p, img.data(), img.size());
  *blob = p;
  *bytes = img.size();
  return BITSMOE_OK;
}

void bitsmoe_blob_free(void* blob) { std::free(blob); }

int bitsmoe_unpack_blob(const void* blob, size_t bytes, bitsmoe_layer_host_out* dst) {
  return bmoe::unpack_image(static_cast<const uint8_t*>(blob), bytes, dst);
}

const char* bitsmoe_strerror(int code) {
  switch (code) {
    case BITSMOE_OK: return "ok";
    case BITSMOE_ERR_INVALID_ARG: return "invalid argument";
    case BITSMOE_ERR_SHAPE: return "unsupported shape";
    case BITSMOE_ERR_UNSUPPORTED_BITS: return "unsupported unit bit-width";
    case BITSMOE_ERR_WORKSPACE_TOO_SMALL: return "workspace too small";
    case BITSMOE_ERR_ALIGNMENT: return "device pointer misaligned";
    case BITSMOE_ERR_CUDA: return "CUDA runtime error";
    case BITSMOE_ERR_OOM: return "out of memory";
    case BITSMOE_ERR_TIMEOUT: return "device wait timed out";
    case BITSMOE_ERR_DEVICE_BOUNDS: return "device bounds check failed";
    case BITSMOE_ERR_BLOB: return "malformed packed blob";
    case BITSMOE_ERR_WORKSPACE_STATE: return "workspace not zero-filled before its first use";
    default: return "unknown error";
  }
}

}  // extern "C"
