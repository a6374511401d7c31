// Per-token compression (Table alg:kvrobin step 7): y = W^T (x - mu), the fused projection +
// Hadamard as one multiply (Sec. 3.4), code = clamp(floor(y / Delta + 2^{b-1}), 0, 2^b - 1),
// packed into code rows (format v1, see include/cobra.h).
//
// compress_kernel  one CTA per (layer, kv head) and chunk of 128-token tiles.  The tile
//                  X [128 x 128] (bf16) is staged in shared memory with cp.async; the fp32
//                  basis is split into 2 or 3 bf16 terms W = W0 + W1 (+ W2) held as MMA B
//                  fragments in shared memory, so Y = X W0 + X W1 (+ X W2) with fp32
//                  accumulation reproduces the fp32 projection; the epilogue quantises and
//                  the CTA packs whole rows with coalesced 32-bit stores.
// append_kernel    one warp per (layer, kv head, sequence): projects the new token in fp32 on
//                  CUDA cores and ORs its codes into the row (other tokens' bits untouched).
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
  int t0, n_tok, chunks;
};

constexpr int kCompressThreads = 256;
constexpr int kWfragBytes = 3 * 16 * 8 * 32 * 8;  // [split][ntile][kstep][lane] uint2
constexpr int kXTileBytes = 128 * 128 * 2;
constexpr int kCodeTileBytes = 128 * 128;
constexpr int kCompressSmem = kWfragBytes + kXTileBytes + kCodeTileBytes;

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\ncp.async.wait_group 0;" ::: "memory");
}
__device__ __forceinline__ void ldmatrix_x4(uint32_t addr, uint32_t& a0, uint32_t& a1, uint32_t& a2, uint32_t& a3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(a0), "=r"(a1), "=r"(a2), "=r"(a3)
               : "r"(addr));
}
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

template <int B>
__device__ void pack_row_tile(const uint8_t* codes, int ldc, int side, int r, uint8_t* row) {
  const int npieces = 8 * (r >> 1);
  for (int idx = threadIdx.x; idx < npieces; idx += kCompressThreads) {
    const int s = idx >> 3, p = idx & 7;
    pack_piece<B>(codes, ldc, side, s, p, reinterpret_cast<uint32_t*>(row + s * 32 * B + p * 4 * B));
  }
}

__global__ void __launch_bounds__(kCompressThreads) compress_kernel(CompressArgs a) {
  extern __shared__ __align__(128) uint8_t smem[];
  uint2* wfrag = reinterpret_cast<uint2*>(smem);
  uint8_t* xt = smem + kWfragBytes;
  uint8_t* codes = xt + kXTileBytes;
  const int head_local = blockIdx.x / a.chunks, chunk = blockIdx.x % a.chunks;
  const int layer = head_local / a.n_kv, kv = head_local % a.n_kv;
  const int hidx = a.head0 + layer * a.layer_stride + kv;
  const HeadEntry he = head_table(a.block)[hidx];
  const int r = he.r, b = he.b;
  const int nrows = (a.n_tok + kRowTokens - 1) / kRowTokens;
  const int ntiles = a.n_seqs * nrows;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t rb = 16u * r * b;
  if (r == 0 || chunk >= ntiles) return;
  const float* pool = param_pool(a.block);
  const float* W = pool + he.w_off;
  const float* wmu = pool + he.wmu_off;
  const int nsplit = b >= 6 ? 3 : 2;
  const int nnt = (r + 7) >> 3;
  // B fragments of the split basis: element (k, n) of (split, nt, ks) = W_split[16 ks + k][8 nt + n]
  for (int idx = tid; idx < nsplit * nnt * 8 * 32; idx += kCompressThreads) {
    const int ln = idx & 31, ks = (idx >> 5) & 7, nt = (idx >> 8) % nnt, sp = idx / (256 * nnt);
    const int j = ln & 3, n = ln >> 2, ch = 8 * nt + n;
    const int ds[4] = {16 * ks + 2 * j, 16 * ks + 2 * j + 1, 16 * ks + 2 * j + 8, 16 * ks + 2 * j + 9};
    float v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      float rem = ch < r ? W[(size_t)ch * kD + ds[u]] : 0.f;
      float part = 0.f;
      for (int q = 0; q <= sp; ++q) {
        part = __bfloat162float(__float2bfloat16_rn(rem));
        rem -= part;
      }
      v[u] = part;
    }
    wfrag[((sp * 16 + nt) * 8 + ks) * 32 + ln] = make_uint2(pack_bf16(v[0], v[1]), pack_bf16(v[2], v[3]));
  }
  const float inv_delta = he.inv_delta, half = (float)(1 << (b - 1));
  const int cmax = (1 << b) - 1;
  const uint32_t xt_base = smem_addr(xt);
  for (int tile = chunk; tile < ntiles; tile += a.chunks) {
    const int seq = tile / nrows, row = tile % nrows;
    const int tok0 = row * kRowTokens;  // relative to t0
    const __nv_bfloat16* xs = a.x + layer * a.sl + seq * a.ss + kv * a.sh;
    __syncthreads();  // previous tile's codes / x tile fully consumed; wfrag written
    for (int idx = tid; idx < 128 * 16; idx += kCompressThreads) {
      const int t = idx >> 4, c = idx & 15;
      const bool valid = tok0 + t < a.n_tok;
      const __nv_bfloat16* src = valid ? xs + (long long)(tok0 + t) * a.st + c * 8 : a.x;
      cp_async16(xt_base + t * 256 + ((c ^ (t & 7)) << 4), src, valid ? 16u : 0u);
    }
    cp_async_wait_all();
    __syncthreads();
    // A fragments of this warp's 16 tokens
    uint32_t af[8][4];
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
      const int t = 16 * warp + (lane & 7) + 8 * ((lane >> 3) & 1);
      const int c = 2 * ks + (lane >> 4);
      ldmatrix_x4(xt_base + t * 256 + ((c ^ (t & 7)) << 4), af[ks][0], af[ks][1], af[ks][2], af[ks][3]);
    }
    const int tA = 16 * warp + (lane >> 2), tB = tA + 8;
    const bool vA = tok0 + tA < a.n_tok, vB = tok0 + tB < a.n_tok;
    for (int nt = 0; nt < nnt; ++nt) {
      float acc[4] = {0.f, 0.f, 0.f, 0.f};
      for (int sp = 0; sp < nsplit; ++sp) {
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
          const uint2 bf = wfrag[((sp * 16 + nt) * 8 + ks) * 32 + lane];
          mma_bf16(acc, af[ks][0], af[ks][1], af[ks][2], af[ks][3], bf.x, bf.y);
        }
      }
      const int ch = 8 * nt + 2 * (lane & 3);
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int c = ch + (u & 1), t = (u < 2) ? tA : tB;
        const bool v = (u < 2) ? vA : vB;
        if (c < r) {
          const float y = acc[u] - wmu[c];
          const float uu = fmaf(y, inv_delta, half);
          int code = (int)floorf(uu);
          code = code < 0 ? 0 : (code > cmax ? cmax : code);
          codes[t * 128 + c] = v ? (uint8_t)code : (uint8_t)0;
        }
      }
    }
    __syncthreads();
    uint8_t* dst = a.cache + row_offset(he.cache_off, rb, seq, (a.t0 >> 7) + row, a.page_table, a.pages_per_seq,
                                        a.rows_per_seq);
    switch (b) {
      case 1: pack_row_tile<1>(codes, 128, a.side, r, dst); break;
      case 2: pack_row_tile<2>(codes, 128, a.side, r, dst); break;
      case 3: pack_row_tile<3>(codes, 128, a.side, r, dst); break;
      case 4: pack_row_tile<4>(codes, 128, a.side, r, dst); break;
      case 5: pack_row_tile<5>(codes, 128, a.side, r, dst); break;
      case 6: pack_row_tile<6>(codes, 128, a.side, r, dst); break;
      case 7: pack_row_tile<7>(codes, 128, a.side, r, dst); break;
      default: pack_row_tile<8>(codes, 128, a.side, r, dst); break;
    }
  }
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
