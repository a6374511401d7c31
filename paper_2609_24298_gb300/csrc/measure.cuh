// Measured per-head distortion tables (App. E, "Exact DP over measured distortion").
//
// For every head, its calibration tokens go through the deployed quantizer once per candidate
// (r, b) and the reconstruction error is measured in the allocator's units:
//   D(r, b) = (1/N) sum_t sum_k omega_k (u_k . (x_t - x^_t))^2,
// omega_k = 1 (MSE objective) or sigma_Q,k^2 (attention-KL objective).  In the eigen
// coordinates c = U^T (x - mu) the error splits exactly into the energy past r,
// sum_{k >= r} omega_k c_k^2, and the quantisation error of the kept coordinates rotated back,
// H_r^T (y - y^) with y = H_r c_r (W = U_r H_r^T, so W^T (x - mu) = H_r c_r).
//
//   coords_kernel   c = (x - mu) U per head, fp32 (one small GEMM per head).
//   measure_kernel  one CTA per (head, r): per token (one warp, 4 coordinates per lane) the
//                   block Walsh-Hadamard transform y = H_r c_r (blocks of the binary digits of
//                   r, largest first, signs on the columns) by butterflies (shuffles for
//                   distances below 32, registers for 32 and 64), then for every b the codes,
//                   the error y - y^, its transform back and the weighted sum.
#pragma once

#include "common.cuh"

namespace cobra {

constexpr int kMeasureMaxR = 65;  // candidate ranks per call
constexpr int kMeasureMaxB = 16;  // candidate bit widths per call

struct MeasureArgs {
  const float* x;        // [n_heads][n_tok][kD] calibration tokens
  const float* U;        // [n_heads][kD * kD] basis, column k = u_k (allocator order)
  const double* lam;     // [n_heads][kD] eigenvalues in the same order
  const double* w;       // [n_heads][kD] allocator weights in the same order (lambda or sigma_Q^2 lambda)
  const float* mu;       // [n_heads][kD]
  const int8_t* signs;   // [n_heads][kD] Hadamard column signs
  float* coords;         // [n_heads][n_tok][kD] workspace: c = (x - mu) U
  double* D;             // [n_heads][n_r][n_b]
  int n_tok, n_r, n_b;
  int r[kMeasureMaxR];
  int b[kMeasureMaxB];
  double L[kMeasureMaxB];  // loading factor of b[j]
};

// c = (x - mu) U for 32 tokens of one head per CTA: the tokens are staged in shared memory,
// U in chunks of 32 rows; thread (token tl, column group kk) computes 16 columns k = kk + 8 m.
constexpr int kCoordTok = 32;
__global__ void __launch_bounds__(256) coords_kernel(MeasureArgs a) {
  __shared__ float xs[kCoordTok][kD + 1];
  __shared__ float us[32][kD + 4];
  const int h = blockIdx.y, t0 = blockIdx.x * kCoordTok, tid = threadIdx.x;
  const int nt = min(kCoordTok, a.n_tok - t0);
  const float* xh = a.x + ((size_t)h * a.n_tok + t0) * kD;
  const float* mu = a.mu + (size_t)h * kD;
  for (int idx = tid; idx < kCoordTok * kD; idx += 256) {
    const int t = idx / kD, i = idx % kD;
    xs[t][i] = t < nt ? xh[(size_t)t * kD + i] - mu[i] : 0.f;
  }
  const int tl = tid >> 3, kk = tid & 7;
  float acc[16];
#pragma unroll
  for (int m = 0; m < 16; ++m) acc[m] = 0.f;
  const float* U = a.U + (size_t)h * kD * kD;
  for (int i0 = 0; i0 < kD; i0 += 32) {
    __syncthreads();  // xs staged / the previous chunk of U consumed
    for (int idx = tid; idx < 32 * kD; idx += 256) {
      const int k = idx / 32, i = idx % 32;  // coalesced along i (column-major U)
      us[i][k] = U[(size_t)k * kD + i0 + i];
    }
    __syncthreads();
    for (int i = 0; i < 32; ++i) {
      const float xv = xs[tl][i0 + i];
#pragma unroll
      for (int m = 0; m < 16; ++m) acc[m] = fmaf(xv, us[i][kk + 8 * m], acc[m]);
    }
  }
  if (tl < nt) {
    float* c = a.coords + ((size_t)h * a.n_tok + t0 + tl) * kD;
#pragma unroll
    for (int m = 0; m < 16; ++m) c[kk + 8 * m] = acc[m];
  }
}

// In-place block Walsh-Hadamard butterflies on a warp's 128-vector (lane holds elements
// lane + 32 m): for every distance d below the element's block size, the pair (k, k ^ d)
// becomes (a + b, a - b) with a the lower index.  bs[m] = block size of element lane + 32 m.
__device__ __forceinline__ void block_wht(float (&v)[4], const int (&bs)[4], int lane) {
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
#pragma unroll
    for (int m = 0; m < 4; ++m) {
      const float o = __shfl_xor_sync(0xffffffffu, v[m], d);
      if (d < bs[m]) v[m] = (lane & d) ? (o - v[m]) : (v[m] + o);
    }
  }
  // distance 32: elements m and m ^ 1; distance 64: m and m ^ 2
#pragma unroll
  for (int dm = 1; dm <= 2; dm <<= 1) {
    float w[4];
#pragma unroll
    for (int m = 0; m < 4; ++m) w[m] = v[m ^ dm];
#pragma unroll
    for (int m = 0; m < 4; ++m)
      if (32 * dm < bs[m]) v[m] = (m & dm) ? (w[m] - v[m]) : (v[m] + w[m]);
  }
}

__global__ void __launch_bounds__(256) measure_kernel(MeasureArgs a) {
  const int h = blockIdx.y, ri = blockIdx.x;
  const int r = a.r[ri];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __shared__ double red[8][kMeasureMaxB + 1];
  // block of each of the lane's elements: binary digits of r, largest first
  int bs[4];
  float sg[4], om[4], inv[4];
  const int8_t* s = a.signs + (size_t)h * kD;
  const double* wt = a.w + (size_t)h * kD;
  const double* lam = a.lam + (size_t)h * kD;
#pragma unroll
  for (int m = 0; m < 4; ++m) {
    const int k = lane + 32 * m;
    int o = 0, size = 0;
    for (int p = 7; p >= 0; --p)
      if (r & (1 << p)) {
        if (k >= o && k < o + (1 << p)) size = 1 << p;
        o += 1 << p;
      }
    bs[m] = size;  // 0 past r
    sg[m] = k < r ? (float)s[k] : 0.f;
    // error weight omega_k = w_k / lambda_k: 1 for the MSE objective, sigma_Q,k^2 for attention-KL
    om[m] = lam[k] > 0.0 ? (float)(wt[k] / lam[k]) : 0.f;
    inv[m] = size > 0 ? rsqrtf((float)size) : 0.f;
  }
  // with unit weights (the MSE objective) the rotation back preserves the norm: the error is
  // summed in the rotated coordinates and the second transform is skipped
  const bool unit_w = __all_sync(0xffffffffu, om[0] == 1.f && om[1] == 1.f && om[2] == 1.f && om[3] == 1.f);
  // Delta per b, as the stored fp32 step: 2 L_b sigma_bar / 2^b, sigma_bar^2 = mean lambda_{<r}
  float delta[kMeasureMaxB], inv_delta[kMeasureMaxB];
  double lsum = 0.0;
  for (int k = 0; k < r; ++k) lsum += a.lam[(size_t)h * kD + k];
  const double sigma = r > 0 ? sqrt(lsum / r) : 0.0;
#pragma unroll
  for (int j = 0; j < kMeasureMaxB; ++j) {
    delta[j] = j < a.n_b ? (float)(2.0 * a.L[j] * sigma / (double)(1 << a.b[j])) : 0.f;
    inv_delta[j] = delta[j] > 0.f ? 1.f / delta[j] : 0.f;
  }

  float acc_trunc = 0.f, acc[kMeasureMaxB];
#pragma unroll
  for (int j = 0; j < kMeasureMaxB; ++j) acc[j] = 0.f;
  for (int t = warp; t < a.n_tok; t += 8) {
    const float* c = a.coords + ((size_t)h * a.n_tok + t) * kD;
    float y[4];
#pragma unroll
    for (int m = 0; m < 4; ++m) {
      const float cv = c[lane + 32 * m];
      if (bs[m] == 0) acc_trunc = fmaf(om[m] * cv, cv, acc_trunc);
      y[m] = cv * sg[m];
    }
    if (r == 0) continue;
    block_wht(y, bs, lane);
#pragma unroll
    for (int m = 0; m < 4; ++m) y[m] *= inv[m];
#pragma unroll
    for (int j = 0; j < kMeasureMaxB; ++j) {
      if (j >= a.n_b) break;
      const int bb = a.b[j];
      const float half = (float)(1 << (bb - 1)), cmax = (float)((1 << bb) - 1), dl = delta[j], il = inv_delta[j];
      float e[4];
#pragma unroll
      for (int m = 0; m < 4; ++m) {
        // (a code may differ from the exact division's at a cell boundary, where both cells
        // leave an error of the same size)
        float code = floorf(fmaf(y[m], il, half));
        code = fminf(fmaxf(code, 0.f), cmax);
        e[m] = bs[m] > 0 ? y[m] - dl * (code - half + 0.5f) : 0.f;
      }
      if (unit_w) {
#pragma unroll
        for (int m = 0; m < 4; ++m) acc[j] = fmaf(e[m], e[m], acc[j]);
        continue;
      }
      // back to the eigen coordinates: H_r^T = diag(s) blockdiag(H_n / sqrt n) (H_n symmetric)
      block_wht(e, bs, lane);
#pragma unroll
      for (int m = 0; m < 4; ++m) {
        const float ek = e[m] * inv[m] * sg[m];
        acc[j] = fmaf(om[m] * ek, ek, acc[j]);
      }
    }
  }
  // reduce over the warp, then over the 8 warps in fp64
#pragma unroll
  for (int o = 16; o; o >>= 1) acc_trunc += __shfl_xor_sync(0xffffffffu, acc_trunc, o);
#pragma unroll
  for (int j = 0; j < kMeasureMaxB; ++j)
#pragma unroll
    for (int o = 16; o; o >>= 1) acc[j] += __shfl_xor_sync(0xffffffffu, acc[j], o);
  if (lane == 0) {
    red[warp][kMeasureMaxB] = acc_trunc;
#pragma unroll
    for (int j = 0; j < kMeasureMaxB; ++j) red[warp][j] = acc[j];
  }
  __syncthreads();
  if (threadIdx.x < a.n_b) {
    const int j = threadIdx.x;
    double tr = 0.0, kept = 0.0;
    for (int w = 0; w < 8; ++w) {
      tr += red[w][kMeasureMaxB];
      kept += red[w][j];
    }
    a.D[((size_t)h * a.n_r + ri) * a.n_b + j] = (tr + kept) / (double)a.n_tok;
  }
}

}  // namespace cobra
