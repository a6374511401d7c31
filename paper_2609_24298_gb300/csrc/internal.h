// Internal layouts shared by the host code and the CUDA kernels of libcobra (not part of
// the public ABI in include/cobra.h).
#pragma once

#include <stddef.h>
#include <stdint.h>

namespace cobra {

constexpr int kD = 128;                 // head dimension
constexpr int kRowTokens = 128;         // tokens per code row
constexpr uint32_t kBlockMagic = 0x52424F43u;  // "COBR"
constexpr uint32_t kWsMagic = 0x53574F43u;     // "COWS"

// Device parameter block: header | head table | float pool.
struct BlockHeader {
  uint32_t magic;
  uint32_t version;
  int32_t n_heads;
  int32_t d;
  uint64_t heads_off;    // bytes from block start
  uint64_t pool_off;     // bytes from block start
  uint64_t pool_floats;
  uint64_t checksum;     // FNV-1a 64 of the whole block with this field zero
  uint64_t reserved[2];
};
static_assert(sizeof(BlockHeader) == 64, "header size");

struct HeadEntry {
  int32_t r, b;
  float delta, inv_delta;
  uint64_t cache_off;  // bytes into the cache buffer
  uint64_t w_off;      // floats into the pool: W, d x r column-major
  uint64_t mu_off;     // floats into the pool: mu, d
  uint64_t wmu_off;    // floats into the pool: W^T mu, r
  uint64_t reserved[2];
};
static_assert(sizeof(HeadEntry) == 64, "head entry size");

// Decode workspace: header | groups | items | head-group table | q~ blocks | partials.
struct WsHeader {
  uint32_t magic;
  uint32_t version;
  int32_t n_groups;
  int32_t n_items;
  int32_t group;      // G
  int32_t n_layers;
  int32_t n_kv;
  int32_t n_seqs;
  uint64_t groups_off, items_off, qt_off, part_off;  // bytes from workspace start
  int32_t part_stride;  // floats per item partial
  int32_t g_stride;     // floats per query head inside a partial: [m, l, -, -, O[0..max_rv)]
  int32_t qt_stride;    // bytes per group q~ block
  int32_t max_rv;
  int32_t max_row_bytes;  // largest K or V code row among the planned heads
  int32_t reserved0;
  uint64_t hg_off;        // int32 [n_layers * n_kv][n_seqs]: group index of (head, seq)
  int32_t reserved[6];
  uint32_t done_ctas;     // scan CTAs that have finished taking items in the running launch
  uint32_t next_item;     // scan work counter: 0 between launches (the scan's last CTA resets it)
};
static_assert(sizeof(WsHeader) == 128, "ws header size");

// A group's chunks write their partials to slots first_item .. first_item + n_items - 1.
struct WsGroup {
  int32_t seq, layer, kv, first_item;
  int32_t n_items, k_head, v_head, reserved;
};
// Work items in the order the scan takes them; slot is the partial the chunk writes.
struct WsItem {
  int32_t group, row_begin, row_end, slot;
};

// q~ block per group: Qsum[8] (fp32, sum of the fp16 hi+lo values per query head),
// scale (fp32, 2^-e), then B fragments [kappa 0..7][ntile 0..1][lane 0..31] of uint2.
constexpr int kQtHeaderBytes = 64;
constexpr int kQtStride = kQtHeaderBytes + 8 * 2 * 32 * 8;

constexpr size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

}  // namespace cobra
