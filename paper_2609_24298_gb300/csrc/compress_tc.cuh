// Per-token compression on the 5th-generation tensor cores (Table alg:kvrobin step 7):
// y = W^T (x - mu) for 128-token tiles, code = clamp(floor(y / Delta + 2^{b-1}), 0, 2^b - 1),
// packed into code rows (format v1, see include/cobra.h).
//
// One CTA per (layer, kv head) and chunk of 128-token tiles, 6 warps:
//   warp 0    TMA producer: each tile X [128 tokens x 128 dims] bf16 arrives as two 64-dim
//             boxes with 128-byte swizzle into a 2-stage shared-memory ring.
//   warp 1    allocates TMEM; one thread issues tcgen05.mma (M = 128 tokens, N = r padded to
//             16, K = 16 per instruction, bf16 inputs, fp32 accumulation in TMEM) against the
//             head's basis, which the CTA splits once into 2 (b <= 5) or 3 (b >= 6) bf16
//             terms W = W0 + W1 (+ W2) held in shared memory in the same swizzled K-major
//             layout: Y = X W0 + X W1 (+ X W2) reproduces the fp32 projection.  Two TMEM
//             accumulators alternate between tiles.
//   warps 2-5 epilogue: each reads its 32 TMEM lanes (tokens), subtracts W^T mu, quantises,
//             writes the codes into a shared tile, and the four warps pack whole code rows
//             with 32-bit stores.
// All waits are bounded; on a timeout the kernel records it in the status word, drains the
// copies and MMAs it issued, frees its TMEM and returns.
#pragma once

#include <cuda.h>

#include "common.cuh"
#include "compress.cuh"

namespace cobra {

constexpr int kTcThreads = 192;
constexpr uint64_t kTcWaitNs = 2000000000ull;  // 2 s
constexpr int kTcEpiWarp0 = 2;
constexpr int kTcTmemCols = 256;           // two accumulators of up to 128 columns
constexpr int kTcXStageBytes = 2 * 16384;  // two 64-dim swizzle atoms of 128 rows
constexpr int kTcCodeLd = 132;             // padded row stride of the code tile (bank spread)
constexpr int kTcWBytes = 3 * 2 * 128 * 128;
constexpr int kTcSmemBytes = 1024 + kTcWBytes + 2 * kTcXStageBytes + 128 * kTcCodeLd + 128 * 4 + 256;

struct TcArgs {
  const unsigned char* block;
  unsigned char* cache;
  const int* page_table;
  int head0, layer_stride, n_kv, side, n_seqs, rows_per_seq, pages_per_seq;
  int t0, n_tok, chunks;
  // tensor-map coordinate slot (1..4) of the head, token, sequence and layer indices
  int slot_head, slot_tok, slot_seq, slot_layer;
};

// ---------------------------------------------------------------------------------------
// PTX wrappers (tcgen05, TMA tensor loads)
// ---------------------------------------------------------------------------------------
__device__ __forceinline__ void tma_load_5d(uint32_t dst, const CUtensorMap* map, const int (&c)[5], uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.5d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4, %5, "
      "%6}], [%7];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c[0]), "r"(c[1]), "r"(c[2]), "r"(c[3]), "r"(c[4]), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void tmem_alloc(uint32_t holder_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(holder_smem), "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void tc_mma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(
          d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void tc_ld16(uint32_t taddr, uint32_t (&v)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]), "=r"(v[8]),
        "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
      : "r"(taddr)
      : "memory");
}
__device__ __forceinline__ void tc_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void named_bar_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

// Shared-memory matrix descriptor of a K-major operand in the 128-byte swizzled canonical
// layout: rows of 128 bytes, 8-row groups 1024 bytes apart (stride byte offset), atoms
// 1024-byte aligned.  Fields: start address >> 4 (bits 0-13), leading byte offset >> 4
// (16-29, unused for this layout), stride byte offset >> 4 (32-45), descriptor version 1
// (46-47), swizzle mode 2 = 128 B (61-63).
__device__ __forceinline__ uint64_t umma_desc_sw128(uint32_t saddr) {
  return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
         ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}
// Instruction descriptor, kind::f16: D fp32 (bits 4-5 = 1), A and B bf16 (bits 7-9 = 1,
// 10-12 = 1), both K-major (bits 15, 16 = 0), N >> 3 (bits 17-22), M >> 4 (bits 24-28).
__device__ __forceinline__ uint32_t umma_idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

__global__ void __launch_bounds__(kTcThreads, 1)
    compress_tc_kernel(const __grid_constant__ CUtensorMap xmap, TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  uint8_t* base = smem_raw + (((raw + 1023u) & ~1023u) - raw);  // 1024-aligned for the swizzle
  uint8_t* wsm = base;                                           // [split][atom][Npad rows][128 B]
  uint8_t* xsm = wsm + kTcWBytes;                                // [stage][atom][128 rows][128 B]
  uint8_t* codes = xsm + 2 * kTcXStageBytes;                     // [128 tokens][kTcCodeLd]
  float* wmu_s = reinterpret_cast<float*>(codes + 128 * kTcCodeLd);
  uint64_t* bars = reinterpret_cast<uint64_t*>(wmu_s + 128);     // x_full[2] x_empty[2] acc_full[2] acc_empty[2] done
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bars + 9);
  int* counters = reinterpret_cast<int*>(tmem_holder + 1);       // [0] tiles issued by TMA, [1] consumed by MMA, [2] fail
  int* epi_ok = counters + 4;                                    // one flag per epilogue warp

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int head_local = blockIdx.x / a.chunks, chunk = blockIdx.x % a.chunks;
  const int layer = head_local / a.n_kv, kv = head_local % a.n_kv;
  const HeadEntry he = head_table(a.block)[a.head0 + layer * a.layer_stride + kv];
  const int r = he.r, b = he.b;
  const int nrows = (a.n_tok + kRowTokens - 1) / kRowTokens;
  const int ntiles = a.n_seqs * nrows;
  if (r == 0 || chunk >= ntiles) return;
  const int my_tiles = (ntiles - chunk + a.chunks - 1) / a.chunks;
  const int npad = (r + 15) & ~15;
  const int nsplit = b >= 6 ? 3 : 2;
  const float* pool = param_pool(a.block);
  const float* W = pool + he.w_off;

  // ---- setup: barriers, TMEM, split basis, W^T mu ----
  if (tid == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_addr(&bars[i]), 1);          // x_full: producer arrive + TMA bytes
      mbar_init(smem_addr(&bars[2 + i]), 1);      // x_empty: MMA commit
      mbar_init(smem_addr(&bars[4 + i]), 1);      // acc_full: MMA commit
      mbar_init(smem_addr(&bars[6 + i]), 4);      // acc_empty: one arrive per epilogue warp
    }
    mbar_init(smem_addr(&bars[8]), 1);            // done: final MMA commit
    counters[0] = counters[1] = counters[2] = 0;
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc(smem_addr(tmem_holder), kTcTmemCols);
  // W split term sp of channel n, dims [64 atom, 64 atom + 64): 8 chunks of 16 bytes per row,
  // chunk c stored at position c ^ (n & 7)
  for (int idx = tid; idx < nsplit * 2 * npad * 8; idx += kTcThreads) {
    const int c = idx & 7, n = (idx >> 3) % npad, atom = (idx / (8 * npad)) & 1, sp = idx / (16 * npad);
    uint32_t packed[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      float v2[2];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int dim = 64 * atom + 8 * c + 2 * e + h;
        float rem = n < r ? W[(size_t)n * kD + dim] : 0.f;
        float part = 0.f;
        for (int q = 0; q <= sp; ++q) {
          part = __bfloat162float(__float2bfloat16_rn(rem));
          rem -= part;
        }
        v2[h] = part;
      }
      packed[e] = pack_bf16(v2[0], v2[1]);
    }
    uint8_t* rowp = wsm + (size_t)sp * 2 * npad * 128 + (size_t)atom * npad * 128 + (size_t)n * 128;
    *reinterpret_cast<uint4*>(rowp + ((c ^ (n & 7)) << 4)) = make_uint4(packed[0], packed[1], packed[2], packed[3]);
  }
  for (int i = tid; i < 128; i += kTcThreads) wmu_s[i] = i < r ? pool[he.wmu_off + i] : 0.f;
  // generic-proxy writes of the basis must be visible to the tensor cores (async proxy)
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;
  const uint32_t bar0 = smem_addr(bars);
  auto bar = [&](int i) { return bar0 + 8u * i; };

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      int issued = 0;
      for (int i = 0; i < my_tiles; ++i) {
        const int st = i & 1;
        if (!mbar_wait_bounded(bar(2 + st), ((i >> 1) & 1) ^ 1, kTcWaitNs)) {
          atomicOr(&g_status, 1u);
          counters[2] = 1;
          break;
        }
        if (counters[2]) break;
        const int tile = chunk + i * a.chunks;
        const int seq = tile / nrows, row = tile % nrows;
        int c[5] = {0, 0, 0, 0, 0};
        c[a.slot_head] = kv;
        c[a.slot_tok] = row * kRowTokens;
        c[a.slot_seq] = seq;
        c[a.slot_layer] = layer;
        mbar_arrive_expect_tx(bar(st), kTcXStageBytes);
        const uint32_t dst = smem_addr(xsm + st * kTcXStageBytes);
        tma_load_5d(dst, &xmap, c, bar(st));
        c[0] = 64;
        tma_load_5d(dst + 16384, &xmap, c, bar(st));
        ++issued;
      }
      counters[0] = issued;
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      const uint32_t idesc = umma_idesc_bf16(128, npad);
      const uint32_t wbase = smem_addr(wsm), xbase = smem_addr(xsm);
      int consumed = 0;
      for (int i = 0; i < my_tiles; ++i) {
        const int st = i & 1, acc = i & 1;
        if (!mbar_wait_bounded(bar(st), (i >> 1) & 1, kTcWaitNs) ||
            !mbar_wait_bounded(bar(6 + acc), ((i >> 1) & 1) ^ 1, kTcWaitNs)) {
          atomicOr(&g_status, 1u);
          counters[2] = 1;
          break;
        }
        if (counters[2]) break;
        ++consumed;
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)(acc * 128);
        for (int sp = 0; sp < nsplit; ++sp)
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            const uint32_t aoff = (uint32_t)((kk >> 2) * 16384 + (kk & 3) * 32);
            const uint32_t boff = (uint32_t)(sp * 2 * npad * 128 + (kk >> 2) * npad * 128 + (kk & 3) * 32);
            tc_mma_bf16(d, umma_desc_sw128(xbase + st * kTcXStageBytes + aoff), umma_desc_sw128(wbase + boff), idesc,
                        (sp > 0 || kk > 0) ? 1u : 0u);
          }
        tc_commit(bar(2 + st));   // X stage free once these MMAs completed
        tc_commit(bar(4 + acc));  // accumulator ready
      }
      counters[1] = consumed;
      tc_commit(bar(8));  // completes when every MMA issued above has completed
      if (!mbar_wait_bounded(bar(8), 0, kTcWaitNs)) atomicOr(&g_status, 1u);
    }
  } else {
    // ---------------- epilogue (warps 2..5) ----------------
    const int q = warp & 3;               // TMEM lane quarter this warp may access
    const int m = 32 * q + lane;          // token row of the tile
    const int et = tid - kTcEpiWarp0 * 32;  // 0..127
    const float inv_delta = he.inv_delta, half = (float)(1 << (b - 1));
    const int cmax = (1 << b) - 1;
    const uint32_t rb = 16u * r * b;
    for (int i = 0; i < my_tiles; ++i) {
      const int acc = i & 1;
      const bool ok = __all_sync(0xffffffffu, mbar_wait_bounded(bar(4 + acc), (i >> 1) & 1, kTcWaitNs));
      if (lane == 0) {
        epi_ok[warp - kTcEpiWarp0] = ok ? 1 : 0;
        if (!ok) {
          atomicOr(&g_status, 1u);
          counters[2] = 1;
        }
      }
      // the four epilogue warps take the same decision from the same flags
      named_bar_sync(1, 128);
      const bool all_ok = epi_ok[0] && epi_ok[1] && epi_ok[2] && epi_ok[3];
      named_bar_sync(1, 128);
      if (!all_ok) break;
      tc_fence_after();
      const int tile = chunk + i * a.chunks;
      const int seq = tile / nrows, row = tile % nrows;
      const bool valid = row * kRowTokens + m < a.n_tok;
      const uint32_t tbase = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(acc * 128);
      for (int c0 = 0; c0 < npad; c0 += 16) {
        uint32_t v[16];
        tc_ld16(tbase + (uint32_t)c0, v);
        tc_wait_ld();
        uint32_t packed[4] = {0u, 0u, 0u, 0u};
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const int col = c0 + e;
          const float y = __uint_as_float(v[e]) - wmu_s[col];
          int code = (int)floorf(fmaf(y, inv_delta, half));
          code = code < 0 ? 0 : (code > cmax ? cmax : code);
          if (!valid || col >= r) code = 0;
          packed[e >> 2] |= (uint32_t)code << (8 * (e & 3));
        }
        uint32_t* dstc = reinterpret_cast<uint32_t*>(codes + m * kTcCodeLd + c0);
#pragma unroll
        for (int e = 0; e < 4; ++e)
          if (c0 + 4 * e < r) dstc[e] = packed[e];
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(6 + acc));
      named_bar_sync(1, 128);
      uint8_t* dst = a.cache + row_offset(he.cache_off, rb, seq, (a.t0 >> 7) + row, a.page_table, a.pages_per_seq,
                                          a.rows_per_seq);
      const int npieces = 4 * r;
      for (int idx = et; idx < npieces; idx += 128) {
        const int s = idx >> 3, p = idx & 7;
        uint32_t* out = reinterpret_cast<uint32_t*>(dst + s * 32 * b + p * 4 * b);
        switch (b) {
          case 1: pack_piece<1>(codes, kTcCodeLd, a.side, s, p, out); break;
          case 2: pack_piece<2>(codes, kTcCodeLd, a.side, s, p, out); break;
          case 3: pack_piece<3>(codes, kTcCodeLd, a.side, s, p, out); break;
          case 4: pack_piece<4>(codes, kTcCodeLd, a.side, s, p, out); break;
          case 5: pack_piece<5>(codes, kTcCodeLd, a.side, s, p, out); break;
          case 6: pack_piece<6>(codes, kTcCodeLd, a.side, s, p, out); break;
          case 7: pack_piece<7>(codes, kTcCodeLd, a.side, s, p, out); break;
          default: pack_piece<8>(codes, kTcCodeLd, a.side, s, p, out); break;
        }
      }
      named_bar_sync(1, 128);  // the code tile is rewritten by the next tile
    }
  }
  // ---- teardown: drain the TMA loads nobody consumed, then free TMEM ----
  __syncthreads();
  if (tid == 0) {
    for (int i = counters[1]; i < counters[0]; ++i)
      if (!mbar_wait_bounded(bar(i & 1), (i >> 1) & 1, kTcWaitNs)) break;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem, kTcTmemCols);
  }
}

}  // namespace cobra
