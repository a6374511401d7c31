// Per-token compression on the 5th-generation tensor cores (Table alg:kvrobin step 7):
// y = W^T (x - mu) for 128-token tiles, code = clamp(floor(y / Delta + 2^{b-1}), 0, 2^b - 1),
// packed into code rows (format v1, see include/cobra.h).
//
// One CTA per (layer, kv head) and chunk of 128-token tiles, 6 warps:
//   warp 0    TMA producer: each tile X [128 tokens x 128 dims] bf16 arrives as two 64-dim
//             boxes with 128-byte swizzle into a 6-stage shared-memory ring.
//   warp 1    allocates TMEM; one thread issues tcgen05.mma computing the transposed
//             projection Y^T = W X^T (M = 128 channels, rows past r zero; N = 128 tokens;
//             K = 16 per instruction; bf16 inputs, fp32 accumulation in TMEM).  The head's
//             fp32 basis is split once per CTA into 2 (b <= 5) or 3 (b >= 6) bf16 terms
//             W = W0 + W1 (+ W2), so W0 X^T + W1 X^T (+ W2 X^T) reproduces the fp32
//             projection.  The terms are the MMAs' A operand in TMEM, so the tensor cores read
//             only X from shared memory.  Two TMEM accumulators alternate between tiles.
//   warps 2-5 write the basis terms into TMEM (a thread per channel), then run the
//             epilogue: a thread owns one channel (its TMEM lane) and reads the 128 token
//             values of its row of Y^T.  Token t's code goes to bits [(t/8) b, (t/8) b + b)
//             of the channel's sub-stream t % 8, which is exactly where format v1 keeps it
//             (K rows: piece t % 8, code rho = t / 8, half = channel parity; V rows: piece
//             4 (channel parity) + (t/2) % 4, rho = t / 8, half = t % 2).  A lane then owns
//             bytes [16 b i, 16 b (i + 1)) of the code row of its channel i: V rows from its
//             own sub-streams, K rows after exchanging half of them with the partner channel.
//             The lanes write their bytes into a shared-memory staging buffer, and after a
//             barrier of the four warps one thread stores the whole row with a bulk copy.
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
// TMEM: two accumulators of 128 columns (tokens), then the basis terms (64 columns each)
constexpr int kTcTmemCols = 512;
constexpr int kTcWCol = 256;
constexpr int kTcXStageBytes = 2 * 16384;  // two 64-dim swizzle atoms of 128 rows
constexpr int kTcStages = 6;               // X ring
constexpr int kTcRowStage = 16 * 128 * 8;  // one code row of the widest head (r = 128, b = 8)
// X ring, then two code-row staging buffers (the bulk store of one tile's row reads its buffer
// while the next tile's row is written into the other)
constexpr int kTcSmemBytes = 1024 + kTcStages * kTcXStageBytes + 2 * kTcRowStage + 256;

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
// D (+)= A B^T, kind::f16 with bf16 inputs: A [M x K] in TMEM (lane = row m, 32-bit column c =
// elements 2c, 2c + 1 of the row, the lower in the low half), B [N x K] K-major in shared memory.
__device__ __forceinline__ void tc_mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                                               uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n" ::"r"(
          d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// 32 consecutive TMEM columns of the warp's 32 lanes: v[j] = column (taddr + j) of this lane
__device__ __forceinline__ void tc_ld32(uint32_t taddr, uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,"
      "%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]), "=r"(v[8]),
        "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]),
        "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]),
        "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(taddr)
      : "memory");
}
// 16 consecutive TMEM columns of the warp's 32 lanes: column (taddr + j) of this lane = v[j]
__device__ __forceinline__ void tc_st32x16(uint32_t taddr, const uint32_t (&v)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(
          taddr),
      "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]),
      "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
      : "memory");
}
__device__ __forceinline__ void tc_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
// Wait for this thread's TMEM loads, with v (the destination of the load in flight) passed
// through the wait, so that no use of v can be scheduled ahead of it.
__device__ __forceinline__ void tc_wait_ld(uint32_t (&v)[32]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(v[0]), "+r"(v[1]), "+r"(v[2]), "+r"(v[3]), "+r"(v[4]), "+r"(v[5]), "+r"(v[6]), "+r"(v[7]),
                 "+r"(v[8]), "+r"(v[9]), "+r"(v[10]), "+r"(v[11]), "+r"(v[12]), "+r"(v[13]), "+r"(v[14]), "+r"(v[15]),
                 "+r"(v[16]), "+r"(v[17]), "+r"(v[18]), "+r"(v[19]), "+r"(v[20]), "+r"(v[21]), "+r"(v[22]),
                 "+r"(v[23]), "+r"(v[24]), "+r"(v[25]), "+r"(v[26]), "+r"(v[27]), "+r"(v[28]), "+r"(v[29]),
                 "+r"(v[30]), "+r"(v[31])
               :
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
// shared -> global bulk store of `bytes` (a multiple of 16, both addresses 16-byte aligned),
// committed as its own bulk group
__device__ __forceinline__ void bulk_store_s2g(void* dst, uint32_t src, uint32_t bytes) {
  asm volatile(
      "cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;\n"
      "cp.async.bulk.commit_group;" ::"l"(dst),
      "r"(src), "r"(bytes)
      : "memory");
}
// wait until at most one bulk group of this thread is still reading its shared-memory source
__device__ __forceinline__ void bulk_store_wait_read_1() {
  asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
}
// wait until every bulk group of this thread has completed
__device__ __forceinline__ void bulk_store_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
// named barrier `id` over the four epilogue warps
__device__ __forceinline__ void tc_epi_sync(int id) {
  asm volatile("bar.sync %0, 128;" ::"r"(id) : "memory");
}
// the same barrier, returning whether `p` holds in all four warps
__device__ __forceinline__ bool tc_epi_all(int id, bool p) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.b32 p, %1, 0;\n bar.red.and.pred q, %2, 128, p;\n selp.u32 %0, 1, 0, q;\n}\n"
      : "=r"(r)
      : "r"((int)p), "r"(id)
      : "memory");
  return r != 0;
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

// Epilogue state of one thread (one channel).
struct TcEpi {
  // u = y inv_delta + cterm with cterm = 2^{b-1} - (W^T mu)_i inv_delta, both scaled by 2^-b
  // (exact): s = u 2^-b
  float inv_s, cterm_s;
  uint32_t top;  // bit pattern of kTcMagic + 2^b - 1
};

// Rounding down without a float-to-integer conversion: for s in [0, 1], the fp32 sum
// kTcMagic + s 2^b rounded toward -inf is kTcMagic + floor(s 2^b) (the spacing of fp32 values
// in [2^23, 2^24) is 1), so its bit pattern is kTcMagicBits + floor(s 2^b).
constexpr float kTcMagic = 12582912.0f;  // 1.5 * 2^23
constexpr uint32_t kTcMagicBits = 0x4B400000u;

// Each code enters its sub-stream word as (kTcMagicBits + code) << off (and, for a code that
// straddles two words, (kTcMagicBits + code) >> (32 - off) in the next one).  The constant
// parts are disjoint from the code bits, so they add up to a fixed sum per word; starting the
// word at minus that sum leaves exactly the codes once all 16 of the sub-stream's codes are in.
template <int B>
__host__ __device__ constexpr uint32_t tc_word_init(int k) {
  uint32_t acc = 0u;
  for (int rho = 0; rho < 16; ++rho) {
    const int pos = rho * B, kk = pos >> 5, off = pos & 31;
    if (kk == k) acc += kTcMagicBits << off;
    if (off + B > 32 && kk + 1 == k) acc += kTcMagicBits >> (32 - off);
  }
  return 0u - acc;
}

// Codes of the 32 tokens 32 c .. 32 c + 31 of this thread's channel into its sub-streams:
// token t -> sub-stream t % 8, bits [(t / 8) B, (t / 8) B + B).
template <int B, int C>
__device__ __forceinline__ void tc_codes32(const uint32_t (&v)[32], const TcEpi& e, uint32_t (&sub)[8][(B + 1) / 2]) {
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    const int t = 32 * C + j, sig = t & 7, pos = (t >> 3) * B;
    // s = clamp(u 2^-b, 0, 1) (NaN -> 0), then kTcMagic + floor(s 2^b), its top clamped at
    // code 2^b - 1: the bits are kTcMagicBits + clamp(floor(u), 0, 2^b - 1)
    const float s = __saturatef(fmaf(__uint_as_float(v[j]), e.inv_s, e.cterm_s));
    const uint32_t c = min(__float_as_uint(__fmaf_rd(s, (float)(1 << B), kTcMagic)), e.top);
    const int k = pos >> 5, off = pos & 31;
    sub[sig][k] += c << off;
    if (off + B > 32) sub[sig][k + 1] += c >> (32 - off);
  }
}

// Code row bytes [16 B i, 16 B (i + 1)) of channel i from the sub-streams (see the header).
// K rows: word w of piece p = halfword w of sub-stream p of channel 2s (low) and of channel
// 2s + 1 (high); lane pairs swap the four pieces the other one writes.  V rows: word w of piece
// 4 (i % 2) + q = halfword w of sub-streams 2q (low) and 2q + 1 (high) of channel i.
template <int B>
__device__ __forceinline__ void tc_row_words(const uint32_t (&sub)[8][(B + 1) / 2], int side, int lane,
                                             uint32_t (&words)[4 * B]) {
  constexpr int NW = (B + 1) / 2;
  const int par = lane & 1;
  if (side == 0) {
    uint32_t got[4][NW];
#pragma unroll
    for (int j = 0; j < 4; ++j)
#pragma unroll
      for (int k = 0; k < NW; ++k) {
        const uint32_t send = par ? sub[j][k] : sub[4 + j][k];
        got[j][k] = __shfl_xor_sync(0xffffffffu, send, 1);
      }
#pragma unroll
    for (int j = 0; j < 4; ++j)
#pragma unroll
      for (int w = 0; w < B; ++w) {
        const uint32_t mine = par ? sub[4 + j][w >> 1] : sub[j][w >> 1];
        const uint32_t lo = par ? got[j][w >> 1] : mine, hi = par ? mine : got[j][w >> 1];
        words[j * B + w] = __byte_perm(lo, hi, (w & 1) ? 0x7632 : 0x5410);
      }
  } else {
#pragma unroll
    for (int q = 0; q < 4; ++q)
#pragma unroll
      for (int w = 0; w < B; ++w)
        words[q * B + w] = __byte_perm(sub[2 * q][w >> 1], sub[2 * q + 1][w >> 1], (w & 1) ? 0x7632 : 0x5410);
  }
}

// The epilogue warps' loop over this CTA's tiles, for bit width B.
template <int B>
__device__ __forceinline__ void tc_epilogue(const TcArgs& a, const HeadEntry& he, const TcEpi& e, int chunk,
                                            int my_tiles, int nrows, uint32_t tmem_q, uint32_t bar_acc_full,
                                            uint32_t bar_acc_empty, uint8_t* rsm, int* fail) {
  constexpr int NW = (B + 1) / 2;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int ch = 32 * (warp & 3) + lane;  // this thread's channel = its TMEM lane
  const uint32_t rb = 16u * he.r * B;
  // the first epilogue thread issues the bulk stores of the code rows
  const bool issuer = threadIdx.x == 32 * kTcEpiWarp0;
  for (int i = 0; i < my_tiles; ++i) {
    const int acc = i & 1;
    const bool ok = __all_sync(0xffffffffu, mbar_wait_bounded(bar_acc_full + 8u * acc, (i >> 1) & 1, kTcWaitNs));
    // the row staging buffer of tile i is free once the bulk store of tile i - 2 has read it
    if (issuer) bulk_store_wait_read_1();
    // every epilogue warp meets here once per tile; a failed wait in any of them stops all four
    if (!tc_epi_all(1, ok)) {
      if (lane == 0 && !ok) {
        atomicOr(&g_status, 1u);
        *fail = 1;
      }
      break;
    }
    tc_fence_after();
    uint32_t sub[8][NW];
#pragma unroll
    for (int s = 0; s < 8; ++s)
#pragma unroll
      for (int k = 0; k < NW; ++k) sub[s][k] = tc_word_init<B>(k);
    const uint32_t tb = tmem_q + (uint32_t)(acc * 128);
    {
      // each load of 32 columns is in flight while the previous 32 are quantised
      uint32_t v0[32], v1[32];
      tc_ld32(tb + 0, v0);
      tc_wait_ld(v0);
      tc_ld32(tb + 32, v1);
      tc_codes32<B, 0>(v0, e, sub);
      tc_wait_ld(v1);
      tc_ld32(tb + 64, v0);
      tc_codes32<B, 1>(v1, e, sub);
      tc_wait_ld(v0);
      tc_ld32(tb + 96, v1);
      tc_codes32<B, 2>(v0, e, sub);
      tc_wait_ld(v1);
      tc_codes32<B, 3>(v1, e, sub);
    }
    // the accumulator can take the next tile's MMAs
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(bar_acc_empty + 8u * acc);
    const int tile = chunk + i * a.chunks;
    const int seq = tile / nrows, row = tile % nrows;
    const int nvalid = min(kRowTokens, a.n_tok - row * kRowTokens);
    if (nvalid < kRowTokens) {
      // tokens past the end are zero bits: sub-stream s keeps the codes rho < ceil((nvalid - s) / 8)
#pragma unroll
      for (int s = 0; s < 8; ++s) {
        const int keep = max(0, min(16, (nvalid - s + 7) >> 3)) * B;
#pragma unroll
        for (int k = 0; k < NW; ++k) {
          const int lo = 32 * k;
          const uint32_t m = keep >= lo + 32 ? 0xffffffffu : (keep <= lo ? 0u : ((1u << (keep - lo)) - 1u));
          sub[s][k] &= m;
        }
      }
    }
    uint32_t words[4 * B];
    tc_row_words<B>(sub, a.side, lane, words);
    uint8_t* stg = rsm + (size_t)(i & 1) * kTcRowStage;
    if (ch < he.r) {
#pragma unroll
      for (int k = 0; k < B; ++k)
        reinterpret_cast<uint4*>(stg + (size_t)ch * 16 * B)[k] =
            make_uint4(words[4 * k], words[4 * k + 1], words[4 * k + 2], words[4 * k + 3]);
    }
    // the generic-proxy writes of the row must be visible to the bulk copy (async proxy)
    fence_proxy_async_smem();
    tc_epi_sync(2);
    if (issuer) {
      uint8_t* dst = a.cache + row_offset(he.cache_off, rb, seq, (a.t0 >> 7) + row, a.page_table, a.pages_per_seq,
                                          a.rows_per_seq);
      bulk_store_s2g(dst, smem_addr(stg), rb);
    }
  }
  // every row written and the staging buffers read before the CTA's shared memory goes away
  if (issuer) bulk_store_wait_all();
}

__global__ void __launch_bounds__(kTcThreads, 1)
    compress_tc_kernel(const __grid_constant__ CUtensorMap xmap, TcArgs a) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  uint8_t* xsm = smem_raw + (((raw + 1023u) & ~1023u) - raw);  // [stage][atom][128 tokens][128 B], 1024-aligned
  uint8_t* rsm = xsm + kTcStages * kTcXStageBytes;  // [2][kTcRowStage] code rows on their way out
  // x_full[kTcStages] x_empty[kTcStages] acc_full[2] acc_empty[2] done w_ready
  uint64_t* bars = reinterpret_cast<uint64_t*>(rsm + 2 * kTcRowStage);
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(bars + 2 * kTcStages + 6);
  int* counters = reinterpret_cast<int*>(tmem_holder + 1);  // [0] tiles issued by TMA, [1] consumed by MMA, [2] fail

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int head_local = blockIdx.x / a.chunks, chunk = blockIdx.x % a.chunks;
  const int layer = head_local / a.n_kv, kv = head_local % a.n_kv;
  const HeadEntry he = head_table(a.block)[a.head0 + layer * a.layer_stride + kv];
  const int r = he.r, b = he.b;
  const int nrows = (a.n_tok + kRowTokens - 1) / kRowTokens;
  const int ntiles = a.n_seqs * nrows;
  if (r == 0 || chunk >= ntiles) return;
  const int my_tiles = (ntiles - chunk + a.chunks - 1) / a.chunks;
  const int nsplit = b >= 6 ? 3 : 2;
  const float* pool = param_pool(a.block);
  const uint32_t bar0 = smem_addr(bars);
  auto bar = [&](int i) { return bar0 + 8u * i; };
  const int XF = 0, XE = kTcStages, AF = 2 * kTcStages, AE = AF + 2, DONE = AF + 4, WREADY = AF + 5;

  // ---- setup: barriers, TMEM ----
  if (tid == 0) {
    for (int i = 0; i < kTcStages; ++i) {
      mbar_init(bar(XF + i), 1);  // producer arrive + TMA bytes
      mbar_init(bar(XE + i), 1);  // MMA commit
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar(AF + i), 1);  // MMA commit
      mbar_init(bar(AE + i), 4);  // one arrive per epilogue warp
    }
    mbar_init(bar(DONE), 1);    // final MMA commit
    mbar_init(bar(WREADY), 4);  // one arrive per epilogue warp once its basis rows are in TMEM
    counters[0] = counters[1] = counters[2] = 0;
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc(smem_addr(tmem_holder), kTcTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      int issued = 0;
      for (int i = 0; i < my_tiles; ++i) {
        const int st = i % kTcStages, ph = (i / kTcStages) & 1;
        if (!mbar_wait_bounded(bar(XE + st), ph ^ 1, kTcWaitNs)) {
          atomicOr(&g_status, 1u);
          counters[2] = 1;
          break;
        }
        if (counters[2]) break;
        const int tile = chunk + i * a.chunks;
        const int seq = tile / nrows, row = tile % nrows;
        int c[5];
        c[0] = 0;
#pragma unroll
        for (int d = 1; d < 5; ++d)
          c[d] = (a.slot_head == d ? kv : 0) + (a.slot_tok == d ? row * kRowTokens : 0) + (a.slot_seq == d ? seq : 0) +
                 (a.slot_layer == d ? layer : 0);
        mbar_arrive_expect_tx(bar(XF + st), kTcXStageBytes);
        const uint32_t dst = smem_addr(xsm + st * kTcXStageBytes);
        tma_load_5d(dst, &xmap, c, bar(XF + st));
        c[0] = 64;
        tma_load_5d(dst + 16384, &xmap, c, bar(XF + st));
        ++issued;
      }
      counters[0] = issued;
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer: Y^T[128 channels][128 tokens] per tile ----------------
    if (lane == 0) {
      const uint32_t idesc = umma_idesc_bf16(128, 128);
      const uint32_t xbase = smem_addr(xsm);
      int consumed = 0;
      const bool w_ok = mbar_wait_bounded(bar(WREADY), 0, kTcWaitNs);
      if (!w_ok) {
        atomicOr(&g_status, 1u);
        counters[2] = 1;
      }
      tc_fence_after();
      for (int i = 0; w_ok && i < my_tiles; ++i) {
        const int st = i % kTcStages, acc = i & 1;
        if (!mbar_wait_bounded(bar(XF + st), (i / kTcStages) & 1, kTcWaitNs) ||
            !mbar_wait_bounded(bar(AE + acc), ((i >> 1) & 1) ^ 1, kTcWaitNs)) {
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
            const uint32_t koff = (uint32_t)((kk >> 2) * 16384 + (kk & 3) * 32);
            tc_mma_bf16_ts(d, tmem + (uint32_t)(kTcWCol + 64 * sp + 8 * kk),
                           umma_desc_sw128(xbase + st * kTcXStageBytes + koff), idesc, (sp > 0 || kk > 0) ? 1u : 0u);
          }
        tc_commit(bar(XE + st));   // X stage free once these MMAs completed
        tc_commit(bar(AF + acc));  // accumulator ready
      }
      counters[1] = consumed;
      tc_commit(bar(DONE));  // completes when every MMA issued above has completed
      if (!mbar_wait_bounded(bar(DONE), 0, kTcWaitNs)) atomicOr(&g_status, 1u);
    }
  } else {
    // ---------------- epilogue (warps 2..5): one channel per thread ----------------
    const int ch = 32 * (warp & 3) + lane;
    const uint32_t tq = tmem + ((uint32_t)(32 * (warp & 3)) << 16);  // this warp's TMEM lane quarter
    // Basis row of channel ch as nsplit bf16 terms, the A operand of the MMAs: TMEM lane ch,
    // column kTcWCol + 64 sp + c holds dims 2c (low half) and 2c + 1 of term sp; rows of
    // channels >= r are zero.
    {
      const float4* wrow = reinterpret_cast<const float4*>(pool + he.w_off + (size_t)(ch < r ? ch : 0) * kD);
#pragma unroll 1
      for (int q = 0; q < 4; ++q) {
        float rem[32];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const float4 f = ch < r ? wrow[8 * q + u] : make_float4(0.f, 0.f, 0.f, 0.f);
          rem[4 * u] = f.x;
          rem[4 * u + 1] = f.y;
          rem[4 * u + 2] = f.z;
          rem[4 * u + 3] = f.w;
        }
#pragma unroll 1
        for (int sp = 0; sp < nsplit; ++sp) {
          uint32_t packed[16];
#pragma unroll
          for (int c = 0; c < 16; ++c) {
            const float p0 = __bfloat162float(__float2bfloat16_rn(rem[2 * c]));
            const float p1 = __bfloat162float(__float2bfloat16_rn(rem[2 * c + 1]));
            rem[2 * c] -= p0;
            rem[2 * c + 1] -= p1;
            packed[c] = pack_bf16(p0, p1);
          }
          tc_st32x16(tq + (uint32_t)(kTcWCol + 64 * sp + 16 * q), packed);
        }
      }
      tc_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(WREADY));
    }
    TcEpi e;
    const float scale = 1.0f / (float)(1 << b);  // a power of two: the scaled values are exact
    e.inv_s = he.inv_delta * scale;
    e.cterm_s = ((float)(1 << (b - 1)) - (ch < r ? pool[he.wmu_off + ch] : 0.f) * he.inv_delta) * scale;
    e.top = kTcMagicBits + (1u << b) - 1u;
    switch (b) {
      case 1: tc_epilogue<1>(a, he, e, chunk, my_tiles, nrows, tq, bar(AF), bar(AE), rsm, &counters[2]); break;
      case 2: tc_epilogue<2>(a, he, e, chunk, my_tiles, nrows, tq, bar(AF), bar(AE), rsm, &counters[2]); break;
      case 3: tc_epilogue<3>(a, he, e, chunk, my_tiles, nrows, tq, bar(AF), bar(AE), rsm, &counters[2]); break;
      case 4: tc_epilogue<4>(a, he, e, chunk, my_tiles, nrows, tq, bar(AF), bar(AE), rsm, &counters[2]); break;
      case 5: tc_epilogue<5>(a, he, e, chunk, my_tiles, nrows, tq, bar(AF), bar(AE), rsm, &counters[2]); break;
      case 6: tc_epilogue<6>(a, he, e, chunk, my_tiles, nrows, tq, bar(AF), bar(AE), rsm, &counters[2]); break;
      case 7: tc_epilogue<7>(a, he, e, chunk, my_tiles, nrows, tq, bar(AF), bar(AE), rsm, &counters[2]); break;
      default: tc_epilogue<8>(a, he, e, chunk, my_tiles, nrows, tq, bar(AF), bar(AE), rsm, &counters[2]); break;
    }
  }
  // ---- teardown: drain the TMA loads nobody consumed, then free TMEM ----
  __syncthreads();
  if (tid == 0) {
    for (int i = counters[1]; i < counters[0]; ++i)
      if (!mbar_wait_bounded(bar(XF + i % kTcStages), (i / kTcStages) & 1, kTcWaitNs)) break;
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
