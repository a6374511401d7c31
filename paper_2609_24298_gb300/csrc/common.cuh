// Device helpers for libcobra's kernels (sm_103a): PTX wrappers and the register-level
// unpacking of packed code pieces into f16 MMA operands.
#pragma once

#include <cuda_fp16.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "internal.h"

namespace cobra {

// ---------------------------------------------------------------------------------------
// status word: bit 0 = a bounded wait expired
// ---------------------------------------------------------------------------------------
__device__ unsigned int g_status;

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Programmatic dependent launch: a kernel launched with programmatic stream serialisation may
// start before the kernel ahead of it in the stream has finished; it calls grid_dep_wait()
// before reading that kernel's results (a no-op for an ordinary launch).  grid_dep_launch()
// lets the dependent kernel be scheduled once every CTA of this grid has called it or exited.
// Every kernel of the library is launched this way and calls grid_dep_wait() on every path
// before it exits, so that the completion of a kernel implies that of all kernels before it
// in the stream: a kernel only ever waits for its direct predecessor.
__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_dep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
// pull one 128-byte line into L2 (no register result, nothing to wait for)
__device__ __forceinline__ void prefetch_l2(const void* p) { asm volatile("prefetch.global.L2 [%0];" ::"l"(p)); }

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ---------------------------------------------------------------------------------------
// mbarrier + bulk async copy (global -> shared, completion counted in bytes)
// ---------------------------------------------------------------------------------------
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_inval(uint32_t bar) {
  asm volatile("mbarrier.inval.shared::cta.b64 [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// Wait for phase `parity` of `bar` to complete, giving up after ~`limit_ns` nanoseconds.
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity, uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t it = 0;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 255) == 255 && globaltimer_ns() - t0 > limit_ns) return false;
  }
}
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(src), "r"(bytes), "r"(bar)
               : "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
// The same operations executed only where `p` holds: every lane of a warp runs the address
// arithmetic and one lane issues, without a divergent branch.
__device__ __forceinline__ void mbar_arrive_expect_tx_if(bool p, uint32_t bar, uint32_t bytes) {
  asm volatile(
      "{\n .reg .pred q;\n setp.ne.b32 q, %2, 0;\n @q mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n}\n" ::"r"(
          bar),
      "r"(bytes), "r"((int)p)
      : "memory");
}
// adds expected bytes to the current phase without arriving (the arrival comes with a later
// arrive.expect_tx on the same barrier)
__device__ __forceinline__ void mbar_expect_tx_if(bool p, uint32_t bar, uint32_t bytes) {
  asm volatile(
      "{\n .reg .pred q;\n setp.ne.b32 q, %2, 0;\n @q mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], %1;\n}\n" ::"r"(
          bar),
      "r"(bytes), "r"((int)p)
      : "memory");
}
__device__ __forceinline__ void bulk_g2s_if(bool p, uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile(
      "{\n .reg .pred q;\n setp.ne.b32 q, %4, 0;\n"
      " @q cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n}\n" ::"r"(dst),
      "l"(src), "r"(bytes), "r"(bar), "r"((int)p)
      : "memory");
}
// One lane's refill of a ring stage with a K row and a V row on one mbarrier, under one
// predicate: the proxy fence (the warp's generic reads of the stage are ordered before the
// async copies that overwrite it), arrive.expect_tx of both sizes, then the two bulk copies
// (a size of 0 skips that copy).
__device__ __forceinline__ void refill_pair_if(bool p, uint32_t bar, uint32_t dst_k, const void* src_k, uint32_t kb,
                                               uint32_t dst_v, const void* src_v, uint32_t vb) {
  asm volatile(
      "{\n .reg .pred q, qk, qv;\n setp.ne.b32 q, %8, 0;\n"
      " setp.ne.and.b32 qk, %3, 0, q;\n setp.ne.and.b32 qv, %6, 0, q;\n"
      " @q fence.proxy.async.shared::cta;\n"
      " @q mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %7;\n"
      " @qk cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%1], [%2], %3, [%0];\n"
      " @qv cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%4], [%5], %6, [%0];\n}\n" ::"r"(bar),
      "r"(dst_k), "l"(src_k), "r"(kb), "r"(dst_v), "l"(src_v), "r"(vb), "r"(kb + vb), "r"((int)p)
      : "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem_if(bool p) {
  asm volatile("{\n .reg .pred q;\n setp.ne.b32 q, %0, 0;\n @q fence.proxy.async.shared::cta;\n}\n" ::"r"((int)p)
               : "memory");
}

// ---------------------------------------------------------------------------------------
// legacy warp-level MMA (operands in registers) and 8x8 transposition
// ---------------------------------------------------------------------------------------
__device__ __forceinline__ void mma_f16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                                        uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void mma_bf16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                                         uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t movmatrix_t(uint32_t x) {
  uint32_t y;
  asm("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
  return y;
}
// 2^x with the SFU's approximate exponential (flush-to-zero; relative error about 2^-22)
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ uint32_t pack_f16(float lo_col, float hi_col) {
  __half2 h = __floats2half2_rn(lo_col, hi_col);  // .x -> low 16 bits
  return *reinterpret_cast<uint32_t*>(&h);
}

// ---------------------------------------------------------------------------------------
// Unpacking one piece (b little-endian words, 32 codes) into 16 f16x2 registers.
//
// Register rho holds code (rho, 0) in its low half and code (rho, 1) in its high half.  The
// code is masked into mantissa bits [k, k+b) of an f16 whose other bits are those of 1.0
// (kOneH2), so each half reads 1 + code * 2^(k-10): one AND/OR with an immediate mask and the
// shared kOneH2 register (plus at most a shift) yields two codes.  The window k depends on
// rho only; the unit offset and the per-window scale 2^(k-10) are removed after the MMA.
// ---------------------------------------------------------------------------------------
constexpr uint32_t kOneH2 = 0x3C003C00u;  // f16 1.0 in both halves

__host__ __device__ constexpr uint32_t pair_mask(int nbits, int k) {
  return (((1u << nbits) - 1u) << k) * 0x00010001u;
}

template <int B>
struct Window {
  // mantissa position used for register rho
  __host__ __device__ static constexpr int k(int rho) {
    if (B == 1) return (rho >= 5 && rho <= 9) ? rho : (rho >= 10 && rho <= 14) ? rho - 5 : (rho <= 4) ? rho + 5 : 9;
    if (B == 2) {
      const int l = rho & 7, o = 2 * l;
      return (l >= 2 && l <= 4) ? o : (l >= 5) ? o - 6 : o + 4;
    }
    return 10 - B;
  }
  // smallest window of this bit width (the reference the per-window scales are taken against)
  __host__ __device__ static constexpr int kmin() { return B == 1 ? 5 : B == 2 ? 4 : 10 - B; }
  // 2^(10-k): turns (value - 1) back into the code
  __host__ __device__ static constexpr float inv_scale(int rho) { return (float)(1 << (10 - k(rho))); }
};

template <int B>
__host__ __device__ __forceinline__ void load_piece(const uint8_t* p, uint32_t (&w)[B]) {
  if constexpr (B % 4 == 0) {
#pragma unroll
    for (int i = 0; i < B / 4; ++i) {
      const uint4 v = reinterpret_cast<const uint4*>(p)[i];
      w[4 * i + 0] = v.x;
      w[4 * i + 1] = v.y;
      w[4 * i + 2] = v.z;
      w[4 * i + 3] = v.w;
    }
  } else if constexpr (B == 2) {
    const uint2 v = *reinterpret_cast<const uint2*>(p);
    w[0] = v.x;
    w[1] = v.y;
  } else {
#pragma unroll
    for (int i = 0; i < B; ++i) w[i] = reinterpret_cast<const uint32_t*>(p)[i];
  }
}

// One register: codes (rho, 0) and (rho, 1) of the piece held in w.  rho is a compile-time
// constant wherever this is called from an unrolled loop; `one` is kOneH2 held in a register.
template <int B>
__host__ __device__ __forceinline__ uint32_t unpack_reg(const uint32_t (&w)[B], int rho, uint32_t one) {
  if constexpr (B == 1) {
    const int k = Window<1>::k(rho);
    const uint32_t x = w[0];
    const uint32_t t = (rho >= 5 && rho <= 9) ? x : (rho >= 10 && rho <= 14) ? (x >> 5) : (rho <= 4) ? (x << 5) : (x >> 6);
    return (t & pair_mask(1, k)) | one;
  } else if constexpr (B == 2) {
    const int l = rho & 7, k = Window<2>::k(rho);
    const uint32_t x = w[rho >> 3];
    const uint32_t t = (l >= 2 && l <= 4) ? x : (l >= 5) ? (x >> 6) : (x << 4);
    return (t & pair_mask(2, k)) | one;
  } else {
    constexpr int k = 10 - B;
    const int x = rho * B, wi = x >> 4, off = x & 15;
    if (off + B <= 16) {
      const uint32_t t = (off >= k) ? (w[wi] >> (off - k)) : (w[wi] << (k - off));
      return (t & pair_mask(B, k)) | one;
    }
    const int nlo = 16 - off;
    const uint32_t lo = w[wi] >> (off - k);
    const uint32_t hi = w[(wi + 1) < B ? wi + 1 : wi] << (k + nlo);
    return (lo & pair_mask(nlo, k)) | (hi & pair_mask(B - nlo, k + nlo)) | one;
  }
}

template <int B>
__host__ __device__ __forceinline__ void unpack_piece(const uint32_t (&w)[B], uint32_t (&o)[16]) {
#pragma unroll
  for (int rho = 0; rho < 16; ++rho) o[rho] = unpack_reg<B>(w, rho, kOneH2);
}

// Words of the piece at p, or zeros when the strip does not exist.
template <int B>
__device__ __forceinline__ void load_piece_or_zero(const uint8_t* p, bool valid, uint32_t (&w)[B]) {
  if (valid) {
    load_piece<B>(p, w);
  } else {
#pragma unroll
    for (int i = 0; i < B; ++i) w[i] = 0u;
  }
}

// 16-byte global -> shared copies that stay in flight until cp_async_wait_all.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\ncp.async.wait_group 0;" ::: "memory");
}

// Rows [0, r) of a basis (fp32, 128 per row, 16-byte aligned) into shared memory with row
// stride ld floats (a multiple of 4); rows [r, 128) are zeroed.  Every copy is issued before
// any is waited for.  The caller synchronises the block before reading.
// issues the copies only; the caller waits with cp_async_wait_all() before reading dst
__device__ __forceinline__ void stage_basis_issue(const float* W, int r, int ld, float* dst) {
  for (int idx = threadIdx.x; idx < 128 * 32; idx += blockDim.x) {
    const int i = idx >> 5, c = idx & 31;
    float* d = dst + (size_t)i * ld + 4 * c;
    if (i < r)
      cp_async16(smem_addr(d), W + (size_t)idx * 4);
    else
      *reinterpret_cast<float4*>(d) = make_float4(0.f, 0.f, 0.f, 0.f);
  }
}
__device__ __forceinline__ void stage_basis(const float* W, int r, int ld, float* dst) {
  stage_basis_issue(W, r, ld, dst);
  cp_async_wait_all();
}

// ---------------------------------------------------------------------------------------
// parameter block access
// ---------------------------------------------------------------------------------------
__device__ __forceinline__ const HeadEntry* head_table(const unsigned char* block) {
  const BlockHeader* h = reinterpret_cast<const BlockHeader*>(block);
  return reinterpret_cast<const HeadEntry*>(block + h->heads_off);
}
__device__ __forceinline__ const float* param_pool(const unsigned char* block) {
  const BlockHeader* h = reinterpret_cast<const BlockHeader*>(block);
  return reinterpret_cast<const float*>(block + h->pool_off);
}

// Byte address of code row `row` of sequence `seq` inside a head region.
__device__ __forceinline__ uint64_t row_offset(uint64_t region, uint32_t row_bytes, int seq, int row,
                                               const int* page_table, int pages_per_seq, int rows_per_seq) {
  long long slot;
  if (page_table)
    slot = 2LL * page_table[(long long)seq * pages_per_seq + (row >> 1)] + (row & 1);
  else
    slot = (long long)seq * rows_per_seq + row;
  return region + (uint64_t)slot * row_bytes;
}

}  // namespace cobra
