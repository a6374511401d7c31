// Code-row packing shared by the compress kernels (format v1, see include/cobra.h), and the
// single-token append (Table alg:kvrobin step 7): y = W^T (x - mu), the fused projection +
// Hadamard as one multiply (Sec. 3.4), code = clamp(floor(y / Delta + 2^{b-1}), 0, 2^b - 1).
//
// append_kernel    one warp per (layer, kv head, sequence): projects the new token in fp32 on
//                  CUDA cores and ORs its codes into the row (other tokens' bits untouched).
// The bulk compress over 128-token tiles runs on the tensor cores (compress_tc.cuh).
#pragma once

#include "common.cuh"

namespace cobra {

struct CompressArgs {
  const unsigned char* block;
  const __nv_bfloat16* x;
  unsigned char* cache;
  const int* page_table;
  const int* pos;
  long long sl, ss, st, sh;
  int head0, layer_stride, n_layers, n_kv, side, n_seqs, rows_per_seq, pages_per_seq;
  int t0, n_tok;
};

__device__ __forceinline__ uint32_t pack_bf16(float lo_col, float hi_col) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo_col, hi_col);
  return *reinterpret_cast<uint32_t*>(&h);
}

// (token, channel) of code (rho, h) in piece p of strip s.
__device__ __forceinline__ void piece_code_coords(int side, int s, int p, int rho, int h, int& t, int& i) {
  const int tau = rho >> 1, u = rho & 1;
  if (side == 0) {
    t = 16 * tau + p + 8 * u;
    i = 2 * s + h;
  } else {
    const int c = p >> 2, j = p & 3;
    t = 16 * tau + 2 * j + 8 * u + h;
    i = 2 * s + c;
  }
}

// Pack one piece (32 codes) from the code tile into B words.
template <int B>
__device__ __forceinline__ void pack_piece(const uint8_t* codes, int ldc, int side, int s, int p, uint32_t* dst) {
  uint32_t w[B];
#pragma unroll
  for (int k = 0; k < B; ++k) w[k] = 0u;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
#pragma unroll
    for (int rho = 0; rho < 16; ++rho) {
      int t, i;
      piece_code_coords(side, s, p, rho, h, t, i);
      const uint32_t c = codes[t * ldc + i];
#pragma unroll
      for (int bit = 0; bit < B; ++bit) {
        const int x = rho * B + bit;
        w[x >> 4] |= ((c >> bit) & 1u) << (16 * h + (x & 15));
      }
    }
  }
#pragma unroll
  for (int k = 0; k < B; ++k) dst[k] = w[k];
}

// a8: single-token append.  One CTA of 8 warps per (layer, kv head): the head's basis is staged
// in shared memory once (row stride kAppendWLd floats, so that a warp's 16-byte row reads are
// conflict-free) and each warp appends the token of one sequence at a time.  The same steps run
// inside the query projection for the K side (both project through W_K), see qproj_kernel.
constexpr int kAppendThreads = 256;
constexpr int kAppendWLd = 132;
__host__ __device__ constexpr size_t append_smem_bytes() {
  return sizeof(float) * ((size_t)kD * kAppendWLd + (size_t)(kAppendThreads / 32) * kD + kD);
}

// The new token and position of the warp's first sequence, loaded before the basis is waited for.
struct AppendNext {
  __nv_bfloat16 x[4];
  int pos;
};
__device__ __forceinline__ AppendNext append_load(const CompressArgs& a, int layer, int kv, int seq) {
  AppendNext n{};
  if (seq < a.n_seqs) {
    const __nv_bfloat16* xp = a.x + layer * a.sl + seq * a.ss + kv * a.sh;
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int k = 0; k < 4; ++k) n.x[k] = xp[lane + 32 * k];
    n.pos = a.pos[seq];
  }
  return n;
}

// Projects, quantises and writes the new token of sequences warp, warp + nwarps, ... of one head
// (he, at (layer, kv)): y = W^T x - W^T mu from the staged basis Ws (row i = channel i, stride
// kAppendWLd) and wmu, codes into the token's bits of its row with atomics (the row's other
// tokens are untouched).  xs: 128 floats of the warp's shared memory; nx: the first sequence's
// token, from append_load.
__device__ __forceinline__ void append_tokens(const CompressArgs& a, const HeadEntry& he, int layer, int kv,
                                              const float* Ws, const float* wmu, float* xs, int warp, int nwarps,
                                              AppendNext nx) {
  const int lane = threadIdx.x & 31;
  const int r = he.r, b = he.b;
  const uint32_t rb = 16u * r * b;
  const float inv_delta = he.inv_delta, half = (float)(1 << (b - 1));
  const int cmax = (1 << b) - 1;
  for (int seq = warp; seq < a.n_seqs; seq += nwarps) {
#pragma unroll
    for (int k = 0; k < 4; ++k) xs[lane + 32 * k] = __bfloat162float(nx.x[k]);
    const int p = nx.pos;
    // the next sequence's token and position, in flight during this one's projection
    nx = append_load(a, layer, kv, seq + nwarps);
    __syncwarp();
    const int row = p >> 7, tt = p & 127;
    const bool in_range = p >= 0 && (a.page_table ? (row >> 1) < a.pages_per_seq : row < a.rows_per_seq);
    if (!in_range) {  // a position past the cache's capacity is never written
      if (lane == 0) atomicOr(&g_status, 2u);
      __syncwarp();
      continue;
    }
    uint8_t* rowp = a.cache + row_offset(he.cache_off, rb, seq, row, a.page_table, a.pages_per_seq, a.rows_per_seq);
    const int tau = tt >> 4, t16 = tt & 15, rho = 2 * tau + (t16 >> 3);
    for (int i = lane; i < r; i += 32) {
      const float* w = Ws + i * kAppendWLd;
      float y = 0.f;
      for (int dd = 0; dd < kD; dd += 4) {
        const float4 wv = *reinterpret_cast<const float4*>(w + dd);
        const float4 xv = *reinterpret_cast<const float4*>(xs + dd);
        y += wv.x * xv.x + wv.y * xv.y + wv.z * xv.z + wv.w * xv.w;
      }
      y -= wmu[i];
      int code = (int)floorf(fmaf(y, inv_delta, half));
      code = code < 0 ? 0 : (code > cmax ? cmax : code);
      int piece, h;
      if (a.side == 0) {
        piece = t16 & 7;
        h = i & 1;
      } else {
        piece = 4 * (i & 1) + ((t16 >> 1) & 3);
        h = t16 & 1;
      }
      uint32_t* words = reinterpret_cast<uint32_t*>(rowp + (i >> 1) * 32 * b + piece * 4 * b);
      const int x0 = rho * b;
      const int w0 = x0 >> 4, o0 = x0 & 15;
      const int n0 = min(b, 16 - o0);
      const uint32_t m0 = ((1u << n0) - 1u) << (16 * h + o0);
      atomicAnd(words + w0, ~m0);
      atomicOr(words + w0, ((uint32_t)code << (16 * h + o0)) & m0);
      if (n0 < b) {
        const uint32_t m1 = ((1u << (b - n0)) - 1u) << (16 * h);
        atomicAnd(words + w0 + 1, ~m1);
        atomicOr(words + w0 + 1, ((uint32_t)code >> n0) << (16 * h) & m1);
      }
    }
    __syncwarp();  // xs is rewritten for the next sequence
  }
}

// The append of (layer, kv head) number `blk` by one CTA of kAppendThreads threads, with
// append_smem_bytes() of shared memory at apsm.  Run by append_kernel and, in the decode step,
// by the V-side CTAs of the query projection's launch.
__device__ __forceinline__ void append_block(const CompressArgs& a, int blk, float* apsm) {
  float* Ws = apsm;                     // [kD][kAppendWLd]
  const int warp = threadIdx.x >> 5;
  float* wmu = Ws + kD * kAppendWLd + (kAppendThreads / 32) * kD;  // W^T mu
  float* xs = Ws + kD * kAppendWLd + warp * kD;
  const int layer = blk / a.n_kv, kv = blk % a.n_kv;
  const HeadEntry he = head_table(a.block)[a.head0 + layer * a.layer_stride + kv];
  if (he.r == 0) {
    grid_dep_wait();
    return;
  }
  const float* pool = param_pool(a.block);
  // the basis and W^T mu (r floats; the pool is padded to 32 floats, so whole 16-byte chunks
  // stay in it) are parameters: their copies start before the wait for the kernel ahead
  if (threadIdx.x < (he.r + 3) / 4)
    cp_async16(smem_addr(wmu + 4 * threadIdx.x), pool + he.wmu_off + 4 * threadIdx.x);
  stage_basis_issue(pool + he.w_off, he.r, kAppendWLd, Ws);
  // the tokens, positions and the cache may be produced or read by the kernels ahead
  grid_dep_wait();
  const AppendNext nx = append_load(a, layer, kv, warp);  // in flight while the basis arrives
  cp_async_wait_all();
  __syncthreads();
  append_tokens(a, he, layer, kv, Ws, wmu, xs, warp, kAppendThreads / 32, nx);
}

__global__ void __launch_bounds__(kAppendThreads) append_kernel(CompressArgs a) {
  extern __shared__ __align__(16) float apsm[];
  grid_dep_launch();
  append_block(a, blockIdx.x, apsm);
}

}  // namespace cobra
