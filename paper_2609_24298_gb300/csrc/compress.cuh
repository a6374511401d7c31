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

// a8: single-token append.  One warp per (layer, kv head, sequence).
__global__ void __launch_bounds__(128) append_kernel(CompressArgs a) {
  __shared__ float xs[4][kD];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long gw = (long long)blockIdx.x * 4 + warp;
  const long long total = (long long)a.n_layers * a.n_kv * a.n_seqs;
  if (gw >= total) return;
  const int seq = (int)(gw % a.n_seqs);
  const int kv = (int)((gw / a.n_seqs) % a.n_kv);
  const int layer = (int)(gw / ((long long)a.n_seqs * a.n_kv));
  const HeadEntry he = head_table(a.block)[a.head0 + layer * a.layer_stride + kv];
  const int r = he.r, b = he.b;
  const __nv_bfloat16* xp = a.x + layer * a.sl + seq * a.ss + kv * a.sh;
#pragma unroll
  for (int k = 0; k < 4; ++k) xs[warp][lane + 32 * k] = __bfloat162float(xp[lane + 32 * k]);
  __syncwarp();
  if (r == 0) return;
  const int p = a.pos[seq];
  const int row = p >> 7, tt = p & 127;
  const bool in_range = p >= 0 && (a.page_table ? (row >> 1) < a.pages_per_seq : row < a.rows_per_seq);
  if (!in_range) {  // a position past the cache's capacity is never written
    if (lane == 0) atomicOr(&g_status, 2u);
    return;
  }
  const uint32_t rb = 16u * r * b;
  uint8_t* rowp = a.cache + row_offset(he.cache_off, rb, seq, row, a.page_table, a.pages_per_seq, a.rows_per_seq);
  const float* pool = param_pool(a.block);
  const float inv_delta = he.inv_delta, half = (float)(1 << (b - 1));
  const int cmax = (1 << b) - 1;
  const int tau = tt >> 4, t16 = tt & 15, rho = 2 * tau + (t16 >> 3);
  for (int i = lane; i < r; i += 32) {
    const float* w = pool + he.w_off + (size_t)i * kD;
    float y = 0.f;
    for (int dd = 0; dd < kD; dd += 4) {
      const float4 wv = *reinterpret_cast<const float4*>(w + dd);
      y += wv.x * xs[warp][dd] + wv.y * xs[warp][dd + 1] + wv.z * xs[warp][dd + 2] + wv.w * xs[warp][dd + 3];
    }
    y -= pool[he.wmu_off + i];
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
}

}  // namespace cobra
