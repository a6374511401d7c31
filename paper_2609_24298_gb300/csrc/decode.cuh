// Decode attention over the packed cache, in rank space (Table alg:kvrobin step 8; App. G).
//
// Three kernels per call:
//   qproj_kernel    q~_g = (Delta_K / sqrt d) log2(e) W_K^T q_g for the G query heads of a
//                   kv head, split into fp16 hi + lo, laid out as MMA B fragments.
//   decode_kernel   persistent warps over work items (token chunks of one (seq, layer, kv-head)).
//                   Each warp streams its chunk's K and V code rows into a private shared-
//                   memory ring with bulk async copies, unpacks codes in registers and runs
//                   f16 mma.sync with fp32 accumulation:
//                     scores  S[t][col] = sum_i code^K[t][i] q~[i][col]   (M = tokens, K = channels)
//                     values  O[i][g]  += sum_t code^V[t][i] P[t][g]      (M = channels, K = tokens)
//                   with an online softmax in base 2 between them.  Writes per-chunk
//                   partials (m, l, sum_t p_t c^V_t).
//   combine_kernel  merges the chunks of each (seq, layer, kv-head), dequantises the rank-space
//                   average and back-projects once: o = mu_V + W_V Delta_V (acc/l - 2^{b-1} + 1/2).
//
// Query heads per lane.  Lane l (j = l % 4) owns NG = G / 4 query heads:
//   G = 4: head j.  Score columns are interleaved (head g hi, head g lo) in one n-tile, so the
//          lane's columns 2j, 2j+1 are the hi and lo parts of head j; the V side's B operand
//          holds (p_j, 0) in columns (2j, 2j+1).
//   G = 8: heads 2j, 2j+1.  Scores use two n-tiles (q~ hi for heads 0..7 | q~ lo for heads
//          0..7), so the lane's columns 2j, 2j+1 are its two heads in both; the V side's B
//          operand holds (p_2j, p_2j+1).
// Either way the probabilities of a 16-token tile sit in the MMA C-fragment layout and one
// movmatrix per 8 tokens turns them into the V side's B fragment.
#pragma once

#include "common.cuh"

namespace cobra {

constexpr int kDecodeWarps = 4;
constexpr int kMaxStages = 8;
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s

struct DecodeArgs {
  const unsigned char* block;
  const unsigned char* cache;
  const int* seq_lens;
  const int* page_table;
  const __nv_bfloat16* q;
  float* out;
  unsigned char* ws;
  long long q_sl, q_ss, o_sl, o_ss;
  int rows_per_seq, pages_per_seq;
  int ring_bytes;  // per-warp staging ring (>= 2 of the largest code rows, multiple of 128)
  uint32_t one;    // kOneH2, passed at run time so that it stays in a register
};

template <int G>
struct Heads {
  static constexpr int NG = G / 4;  // query heads per lane
  static constexpr int NTK = G / 4; // score n-tiles
  // query head of score column n in n-tile nt, and whether that column holds the lo part
  __host__ __device__ static constexpr int col_head(int nt, int n) { return G == 4 ? n >> 1 : n; }
  __host__ __device__ static constexpr int col_lo(int nt, int n) { return G == 4 ? (n & 1) : nt; }
  // the lane's u-th query head (j = lane % 4)
  __device__ static int head(int j, int u) { return G == 4 ? j : 2 * j + u; }
};

// ---------------------------------------------------------------------------------------
// Per-head kernels (query projection, combine): one CTA of 256 threads per (layer, kv head),
// looping over the sequences 32 query vectors at a time, with the head's basis staged in
// shared memory once.  The workspace's head-group table gives the group of (head, seq).
// ---------------------------------------------------------------------------------------
constexpr int kHeadThreads = 256;
constexpr int kVecPass = 32;  // query vectors (sequences x G) per pass
constexpr int kWLd = 132;     // padded row stride (floats) of a staged basis: conflict-free row reads
constexpr int kZLd = 36;      // row stride of the transposed rank-space averages

__host__ __device__ constexpr size_t qproj_smem_bytes() {
  return sizeof(float) * ((size_t)kD * kWLd + (size_t)kVecPass * kD + (size_t)kVecPass * kWLd);
}
constexpr int kWtChunk = 64;  // chunk weights held in shared memory per vector and round
__host__ __device__ constexpr size_t combine_smem_bytes() {
  return sizeof(float) * ((size_t)kD * kD + (size_t)kD * kZLd + kD + (size_t)kVecPass * kWtChunk);
}

// ---------------------------------------------------------------------------------------
// a4: query projection
//   q~_g = (Delta_K / sqrt d) log2(e) W_K^T q_g per query head, scaled by a power of two so
//   that max |q~| of the group lands in [256, 512), split into fp16 hi + lo and laid out as
//   the scan's MMA B fragments; Qsum_g = sum over channels of the fed hi + lo values.
// ---------------------------------------------------------------------------------------
template <int G>
__global__ void __launch_bounds__(kHeadThreads) qproj_kernel(DecodeArgs a) {
  constexpr int NTK = Heads<G>::NTK, SPP = kVecPass / G;
  extern __shared__ __align__(16) float qsm[];
  float* Ws = qsm;                  // [kD][kWLd]   W_K row i = channel i
  float* Qs = Ws + kD * kWLd;       // [kVecPass][kD] queries of this pass (fp32)
  float* Os = Qs + kVecPass * kD;   // [kVecPass][kWLd] scaled q~ of this pass
  const WsHeader* wh = reinterpret_cast<const WsHeader*>(a.ws);
  const WsGroup* groups = reinterpret_cast<const WsGroup*>(a.ws + wh->groups_off);
  const int S = wh->n_seqs;
  const int* hg = reinterpret_cast<const int*>(a.ws + wh->hg_off) + (size_t)blockIdx.x * S;
  const WsGroup g0 = groups[hg[0]];
  const HeadEntry hk = head_table(a.block)[g0.k_head];
  const float* pool = param_pool(a.block);
  const int r = hk.r, layer = g0.layer, kv = g0.kv;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const float scale = hk.delta * 0.088388347648318440f * 1.4426950408889634f;  // Delta/sqrt(128)*log2(e)
  stage_basis(pool + hk.w_off, r, kWLd, Ws);
  for (int s0 = 0; s0 < S; s0 += SPP) {
    const int ns = min(SPP, S - s0), nv = ns * G;
    __syncthreads();  // basis staged; the previous pass is done with Qs and Os
    // queries are only 2-byte aligned in general: element loads, all issued together
#pragma unroll 16
    for (int idx = tid; idx < nv * kD; idx += kHeadThreads) {
      const int v = idx / kD, d = idx % kD;
      const __nv_bfloat16* qp = a.q + layer * a.q_sl + (long long)(s0 + v / G) * a.q_ss + (long long)(kv * G + v % G) * kD;
      Qs[v * kD + d] = __bfloat162float(qp[d]);
    }
    __syncthreads();
    // warp w: vectors 4w..4w+3; lane: channels lane + 32c
    const int v0 = 4 * warp;
    if (v0 < nv) {
      float acc[4][4];
#pragma unroll
      for (int c = 0; c < 4; ++c)
#pragma unroll
        for (int v = 0; v < 4; ++v) acc[c][v] = 0.f;
#pragma unroll 4
      for (int d = 0; d < kD; d += 4) {
        float4 w[4], q[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) w[c] = *reinterpret_cast<const float4*>(Ws + (lane + 32 * c) * kWLd + d);
#pragma unroll
        for (int v = 0; v < 4; ++v) q[v] = *reinterpret_cast<const float4*>(Qs + (v0 + v) * kD + d);
#pragma unroll
        for (int c = 0; c < 4; ++c)
#pragma unroll
          for (int v = 0; v < 4; ++v)
            acc[c][v] += w[c].x * q[v].x + w[c].y * q[v].y + w[c].z * q[v].z + w[c].w * q[v].w;
      }
#pragma unroll
      for (int c = 0; c < 4; ++c)
#pragma unroll
        for (int v = 0; v < 4; ++v) Os[(v0 + v) * kWLd + lane + 32 * c] = acc[c][v] * scale;
    }
    __syncthreads();
    // per sequence (one warp each): power-of-two scale, hi/lo split, Qsum, B fragments
    for (int sl = warp; sl < ns; sl += kHeadThreads / 32) {
      const float* o = Os + sl * G * kWLd;
      float amax = 0.f;
      for (int i = lane; i < r; i += 32)
#pragma unroll
        for (int g = 0; g < G; ++g) amax = fmaxf(amax, fabsf(o[g * kWLd + i]));
#pragma unroll
      for (int m = 16; m; m >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, m));
      int e = 0;
      if (amax > 0.f) {
        int ex;
        frexpf(amax, &ex);  // amax = m 2^ex, m in [0.5, 1)
        e = 9 - ex;
      }
      const float up = ldexpf(1.f, e);
      unsigned char* qt = a.ws + wh->qt_off + (size_t)hg[s0 + sl] * wh->qt_stride;
      float* qhdr = reinterpret_cast<float*>(qt);
#pragma unroll
      for (int g = 0; g < G; ++g) {
        float sum = 0.f;
        for (int i = lane; i < r; i += 32) {
          const float x = o[g * kWLd + i] * up;
          const __half h = __float2half_rn(x);
          const __half l = __float2half_rn(x - __half2float(h));
          sum += __half2float(h) + __half2float(l);
        }
#pragma unroll
        for (int m = 16; m; m >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, m);
        if (lane == 0) qhdr[g] = sum;
      }
      if (lane == 0) qhdr[8] = ldexpf(1.f, -e);
      // element (k, n) of fragment (kappa, nt) = hi or lo part of q~ of channel 16 kappa + k
      // for the query head of column n (see Heads)
      uint2* frag = reinterpret_cast<uint2*>(qt + kQtHeaderBytes);
      for (int idx = lane; idx < 8 * NTK * 32; idx += 32) {
        const int fl = idx & 31, nt = (idx >> 5) % NTK, kap = idx / (32 * NTK);
        const int j = fl & 3, n = fl >> 2;
        const int g = Heads<G>::col_head(nt, n), lo = Heads<G>::col_lo(nt, n);
        float e4[4];
        const int ks[4] = {2 * j, 2 * j + 1, 2 * j + 8, 2 * j + 9};
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int ch = 16 * kap + ks[u];
          float v = 0.f;
          if (ch < r) {
            const float x = o[g * kWLd + ch] * up;
            const float h = __half2float(__float2half_rn(x));
            v = lo ? (x - h) : h;
          }
          e4[u] = v;
        }
        frag[(kap * 2 + nt) * 32 + fl] = make_uint2(pack_f16(e4[0], e4[1]), pack_f16(e4[2], e4[3]));
      }
    }
  }
}

// ---------------------------------------------------------------------------------------
// a5 + a6: chunked rank-space scan
//
// Per warp: running max m, sum l and offset correction c per owned query head in registers;
// the rank-space value accumulators (the lane's C-fragment entries of O) live in the warp's
// shared memory and are rescaled only when the running max moves.  Loops over k-tiles (K
// side) and channel tiles (V side) stay rolled to keep each (b_K, b_V) variant's code small;
// only the 8 token tiles of a row are unrolled.
// ---------------------------------------------------------------------------------------
template <int G>
struct WarpState {
  static constexpr int NG = G / 4;
  float m[NG], l[NG], c[NG];
};

// accumulator floats per (channel tile, lane): the live C-fragment entries of the V MMA
template <int G>
struct OAcc {
  static constexpr int N = G == 4 ? 2 : 4;  // G = 4: columns 2j only; G = 8: both columns
};

// K side: scores of one code row for the lane's query heads, s[8][NG][2]
// (token t0 = 16 tau + lane/4 in [..][..][0], t1 = t0 + 8 in [..][..][1]), log2 units.
template <int G, int B>
__device__ __forceinline__ void k_row_scores(const uint8_t* stage, int rk, const uint2* bfrag,
                                             const float (&qsum)[G / 4], float qscale, uint32_t one,
                                             float (&s)[8][G / 4][2]) {
  constexpr int NTK = Heads<G>::NTK, NG = Heads<G>::NG;
  const int lane = threadIdx.x & 31;
  float acc[8][NTK][4];
#pragma unroll
  for (int t = 0; t < 8; ++t)
#pragma unroll
    for (int nt = 0; nt < NTK; ++nt) acc[t][nt][0] = acc[t][nt][1] = acc[t][nt][2] = acc[t][nt][3] = 0.f;
  const int P = rk >> 1;
  const int nfull = P >> 3, nk = (P + 7) >> 3;
  // lane's pieces: strips 8 kappa + (lane & 3) and + 4, piece lane >> 2
  const uint8_t* pa = stage + (lane & 3) * 32 * B + (lane >> 2) * 4 * B;
  const uint2* bq = bfrag + lane;
  auto tile = [&](bool check, int kap) {
    // channels past r (a partial last k-tile) multiply q~ = 0, so their operand values only
    // need to be finite; the words are zeroed rather than read past the row
    uint32_t wa[B], wb[B];
    if (check) {
      const int sA = 8 * kap + (lane & 3);
      load_piece_or_zero<B>(pa, sA < P, wa);
      load_piece_or_zero<B>(pa + 4 * 32 * B, sA + 4 < P, wb);
    } else {
      load_piece<B>(pa, wa);
      load_piece<B>(pa + 4 * 32 * B, wb);
    }
    uint2 bf[NTK];
#pragma unroll
    for (int nt = 0; nt < NTK; ++nt) bf[nt] = bq[nt * 32];
#pragma unroll
    for (int t = 0; t < 8; ++t) {
      const uint32_t a0 = unpack_reg<B>(wa, 2 * t, one), a1 = unpack_reg<B>(wa, 2 * t + 1, one);
      const uint32_t a2 = unpack_reg<B>(wb, 2 * t, one), a3 = unpack_reg<B>(wb, 2 * t + 1, one);
#pragma unroll
      for (int nt = 0; nt < NTK; ++nt) mma_f16(acc[t][nt], a0, a1, a2, a3, bf[nt].x, bf[nt].y);
    }
    pa += 8 * 32 * B;
    bq += 2 * 32;
  };
#pragma unroll 1
  for (int kap = 0; kap < nfull; ++kap) tile(false, kap);
  if (nk > nfull) tile(true, nfull);
  // acc = Qsum + 2^(k-10) * sum_i q~_i code_i, Qsum = sum of the q~ fed to the MMA.  b >= 3
  // uses one window for every register, so Qsum shifts every token's score alike and softmax
  // ignores it; b = 1, 2 mix windows, so Qsum is removed before the per-token rescale.
#pragma unroll
  for (int t = 0; t < 8; ++t) {
    const float sc0 = qscale * Window<B>::inv_scale(2 * t), sc1 = qscale * Window<B>::inv_scale(2 * t + 1);
#pragma unroll
    for (int u = 0; u < NG; ++u) {
      // hi + lo parts of the u-th head: G = 4 -> columns (2j, 2j+1) of n-tile 0;
      // G = 8 -> column 2j + u of n-tiles 0 and 1
      const float v0 = G == 4 ? acc[t][0][0] + acc[t][0][1] : acc[t][0][u] + acc[t][NTK - 1][u];
      const float v1 = G == 4 ? acc[t][0][2] + acc[t][0][3] : acc[t][0][2 + u] + acc[t][NTK - 1][2 + u];
      if constexpr (B <= 2) {
        s[t][u][0] = (v0 - qsum[u]) * sc0;
        s[t][u][1] = (v1 - qsum[u]) * sc1;
      } else {
        s[t][u][0] = v0 * sc0;
        s[t][u][1] = v1 * sc1;
      }
    }
  }
}

// V side: add one code row's rank-space contribution into the shared-memory accumulators.
template <int G, int B>
__device__ __forceinline__ void v_row_accumulate(const uint8_t* stage, int rv, const uint32_t (&bv)[8][2],
                                                 uint32_t one, float* osm) {
  constexpr int NO = OAcc<G>::N;
  const int lane = threadIdx.x & 31;
  const int P = rv >> 1;
  const int nfull = P >> 3, nmu = (P + 7) >> 3;
  // lane's pieces: strips 8 mu + (lane >> 3) and + 4, piece lane & 7
  const uint8_t* pa = stage + (lane >> 3) * 32 * B + (lane & 7) * 4 * B;
  float* o = osm + lane * NO;
  auto tile = [&](bool check, int mu) {
    // rows for channels past r are never written out, so their operand values only need to
    // be finite
    uint32_t wa[B], wb[B];
    if (check) {
      const int sA = 8 * mu + (lane >> 3);
      load_piece_or_zero<B>(pa, sA < P, wa);
      load_piece_or_zero<B>(pa + 4 * 32 * B, sA + 4 < P, wb);
    } else {
      load_piece<B>(pa, wa);
      load_piece<B>(pa + 4 * 32 * B, wb);
    }
    // fresh accumulators per row: the running sums in shared memory are dominated by the unit
    // code offsets, so they are only ever updated with round-to-nearest fp32 adds
    float d[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
    for (int t = 0; t < 8; ++t) {
      const uint32_t a0 = unpack_reg<B>(wa, 2 * t, one), a1 = unpack_reg<B>(wb, 2 * t, one);
      const uint32_t a2 = unpack_reg<B>(wa, 2 * t + 1, one), a3 = unpack_reg<B>(wb, 2 * t + 1, one);
      mma_f16(d[t & 1], a0, a1, a2, a3, bv[t][0], bv[t][1]);
    }
    if constexpr (NO == 2) {
      float2 v = *reinterpret_cast<float2*>(o);
      v.x += d[0][0] + d[1][0];
      v.y += d[0][2] + d[1][2];
      *reinterpret_cast<float2*>(o) = v;
    } else {
      float4 v = *reinterpret_cast<float4*>(o);
      v.x += d[0][0] + d[1][0];
      v.y += d[0][1] + d[1][1];
      v.z += d[0][2] + d[1][2];
      v.w += d[0][3] + d[1][3];
      *reinterpret_cast<float4*>(o) = v;
    }
    pa += 8 * 32 * B;
    o += 32 * NO;
  };
#pragma unroll 1
  for (int mu = 0; mu < nfull; ++mu) tile(false, mu);
  if (nmu > nfull) tile(true, nfull);
}

template <int G>
__device__ __forceinline__ void k_row_dispatch(int b, const uint8_t* stage, int rk, const uint2* bfrag,
                                               const float (&qsum)[G / 4], float qscale, uint32_t one,
                                               float (&s)[8][G / 4][2]) {
  switch (b) {
    case 1: k_row_scores<G, 1>(stage, rk, bfrag, qsum, qscale, one, s); break;
    case 2: k_row_scores<G, 2>(stage, rk, bfrag, qsum, qscale, one, s); break;
    case 3: k_row_scores<G, 3>(stage, rk, bfrag, qsum, qscale, one, s); break;
    case 4: k_row_scores<G, 4>(stage, rk, bfrag, qsum, qscale, one, s); break;
    case 5: k_row_scores<G, 5>(stage, rk, bfrag, qsum, qscale, one, s); break;
    case 6: k_row_scores<G, 6>(stage, rk, bfrag, qsum, qscale, one, s); break;
    case 7: k_row_scores<G, 7>(stage, rk, bfrag, qsum, qscale, one, s); break;
    default: k_row_scores<G, 8>(stage, rk, bfrag, qsum, qscale, one, s); break;
  }
}

template <int G>
__device__ __forceinline__ void v_row_dispatch(int b, const uint8_t* stage, int rv, const uint32_t (&bv)[8][2],
                                               uint32_t one, float* osm) {
  switch (b) {
    case 1: v_row_accumulate<G, 1>(stage, rv, bv, one, osm); break;
    case 2: v_row_accumulate<G, 2>(stage, rv, bv, one, osm); break;
    case 3: v_row_accumulate<G, 3>(stage, rv, bv, one, osm); break;
    case 4: v_row_accumulate<G, 4>(stage, rv, bv, one, osm); break;
    case 5: v_row_accumulate<G, 5>(stage, rv, bv, one, osm); break;
    case 6: v_row_accumulate<G, 6>(stage, rv, bv, one, osm); break;
    case 7: v_row_accumulate<G, 7>(stage, rv, bv, one, osm); break;
    default: v_row_accumulate<G, 8>(stage, rv, bv, one, osm); break;
  }
}

template <int G>
__device__ __forceinline__ size_t decode_osm_bytes() {
  return (size_t)8 * 32 * OAcc<G>::N * sizeof(float);
}

// Online softmax of one row's scores (base 2) and the V-side MMA operands.  VC is the V bit
// width's window class: 0 = one window for every register (b >= 3), 1 or 2 = the b = 1 / b = 2
// windows.  V codes read 1 + code * 2^(k-10) with a per-register window k, so each token's
// probability is fed to the MMA pre-scaled by 2^(kmin - k) (folded into the exponent): the
// products then carry the single scale 2^(kmin-10), and the unit offsets add up to the plain
// sum of the fed values, accumulated in c.  Every fed value is rounded to fp16 once and the
// same rounded value enters l, c and the MMA, so the weights stay exactly normalised.
template <int VC>
struct VWin {
  static constexpr int B = VC == 0 ? 3 : VC;
  __device__ static constexpr float shift(int rho) {  // kmin - k (<= 0)
    return VC == 0 ? 0.f : (float)(Window<B>::kmin() - Window<B>::k(rho));
  }
  __device__ static constexpr float unshift(int rho) {  // 2^(k - kmin)
    return VC == 0 ? 1.f : (float)(1 << (Window<B>::k(rho) - Window<B>::kmin()));
  }
};

template <int G, int VC>
__device__ __forceinline__ void row_softmax(float (&s)[8][G / 4][2], WarpState<G>& st, float (&alpha)[G / 4],
                                            bool& rescale, uint32_t (&bv)[8][2]) {
  constexpr int NG = G / 4;
  float pf[8][NG][2];
#pragma unroll
  for (int u = 0; u < NG; ++u) {
    float mx = -INFINITY;
#pragma unroll
    for (int t = 0; t < 8; ++t) mx = fmaxf(mx, fmaxf(s[t][u][0], s[t][u][1]));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
    const float mnew = fmaxf(st.m[u], mx);
    alpha[u] = ex2_approx(st.m[u] - mnew);
    rescale |= (mnew != st.m[u]);
    st.m[u] = mnew;
    float ls = 0.f, cs = 0.f;
#pragma unroll
    for (int t = 0; t < 8; ++t) {
      const float e0 = s[t][u][0] - mnew + VWin<VC>::shift(2 * t);
      const float e1 = s[t][u][1] - mnew + VWin<VC>::shift(2 * t + 1);
      const float2 q = __half22float2(__floats2half2_rn(ex2_approx(e0), ex2_approx(e1)));
      pf[t][u][0] = q.x;
      pf[t][u][1] = q.y;
      if constexpr (VC == 0) {
        ls += q.x + q.y;
      } else {
        ls += q.x * VWin<VC>::unshift(2 * t) + q.y * VWin<VC>::unshift(2 * t + 1);
        cs += q.x + q.y;
      }
    }
    st.l[u] = st.l[u] * alpha[u] + ls;
    st.c[u] = st.c[u] * alpha[u] + cs;
  }
  // B fragments of the V side: the 16 x 8 probability tile of token tile t in C-fragment
  // layout (row t0 or t1, columns 2j, 2j+1), transposed by movmatrix.  The fp16 values are
  // exact (they were rounded above).
#pragma unroll
  for (int t = 0; t < 8; ++t) {
    const float c0 = pf[t][0][0], c1 = NG == 2 ? pf[t][NG - 1][0] : 0.f;
    const float c2 = pf[t][0][1], c3 = NG == 2 ? pf[t][NG - 1][1] : 0.f;
    bv[t][0] = movmatrix_t(pack_f16(c0, c1));
    bv[t][1] = movmatrix_t(pack_f16(c2, c3));
  }
}

template <int G>
__global__ void __launch_bounds__(kDecodeWarps * 32, 4) decode_kernel(DecodeArgs a) {
  constexpr int NG = G / 4, NO = OAcc<G>::N;
  extern __shared__ __align__(128) uint8_t smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int ring_bytes = a.ring_bytes;
  const size_t warp_bytes = (size_t)ring_bytes + decode_osm_bytes<G>();
  uint8_t* ring = smem + (size_t)warp * warp_bytes;
  float* osm = reinterpret_cast<float*>(ring + ring_bytes);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + (size_t)kDecodeWarps * warp_bytes) + warp * kMaxStages;
  if (lane == 0) {
    for (int i = 0; i < kMaxStages; ++i) mbar_init(smem_addr(&bars[i]), 1);
    fence_mbar_init();
  }
  __syncwarp();

  const WsHeader* wh = reinterpret_cast<const WsHeader*>(a.ws);
  const WsGroup* groups = reinterpret_cast<const WsGroup*>(a.ws + wh->groups_off);
  const WsItem* items = reinterpret_cast<const WsItem*>(a.ws + wh->items_off);
  const HeadEntry* heads = head_table(a.block);
  float* parts = reinterpret_cast<float*>(a.ws + wh->part_off);
  const int n_items = wh->n_items;
  const int gstride = wh->g_stride, pstride = wh->part_stride;
  uint32_t phase_bits = 0;  // parity of the next wait per barrier
  bool failed = false;
  int outstanding = 0;      // loads issued but not yet waited for
  int wait_stage = 0, nstage = 2;

  // work items are taken in plan order from a shared counter, so that warps that finish early
  // take more (the items' costs differ with the heads' bit widths)
  unsigned int* next_item = const_cast<unsigned int*>(&wh->next_item);
  auto take = [&]() -> int {
    int v = 0;
    if (lane == 0) v = (int)atomicAdd(next_item, 1u);
    return __shfl_sync(0xffffffffu, v, 0);
  };
  for (int item = take(); item < n_items && !failed; item = take()) {
    const WsItem it = items[item];
    const WsGroup gr = groups[it.group];
    const int kr = heads[gr.k_head].r, kb = heads[gr.k_head].b, vr = heads[gr.v_head].r, vb = heads[gr.v_head].b;
    const uint64_t koff = heads[gr.k_head].cache_off, voff = heads[gr.v_head].cache_off;
    const int T = a.seq_lens[gr.seq];
    const int rows_valid = (T + kRowTokens - 1) / kRowTokens;
    const int row0 = it.row_begin, row1 = min(it.row_end, rows_valid);
    float* part = parts + (size_t)item * pstride;
    const uint32_t rbk = kr > 0 ? 16u * kr * kb : 0u, rbv = vr > 0 ? 16u * vr * vb : 0u;
    // this item's stages: as many buffers of its largest row as the ring holds (every load of
    // the previous item has been consumed, so the ring is free)
    const int stage_bytes = (int)((max(max(rbk, rbv), 16u) + 127u) & ~127u);
    nstage = min(kMaxStages, ring_bytes / stage_bytes);
    wait_stage = 0;
    if (nstage < 2) {
      // a row that does not fit the staging buffer is never copied; report and leave an
      // empty chunk (m = -inf, l = 0)
      if (lane == 0) atomicOr(&g_status, 2u);
      if (lane < G) {
        part[lane * gstride + 0] = -INFINITY;
        part[lane * gstride + 1] = 0.f;
      }
      continue;
    }
    WarpState<G> st;
#pragma unroll
    for (int u = 0; u < NG; ++u) {
      st.m[u] = -INFINITY;
      st.l[u] = 0.f;
      st.c[u] = 0.f;
    }
    const int nmu = ((vr >> 1) + 7) >> 3;
    for (int k = 0; k < nmu * NO; ++k) osm[k * 32 + lane] = 0.f;
    // V window class (see row_softmax) and the factor 2^(10 - kmin) that turns the fed
    // products back into codes
    const int vc = (vr > 0 && vb <= 2) ? vb : 0;
    const float vout = vr == 0 ? 0.f : (float)(1 << (vb == 1 ? 5 : vb == 2 ? 6 : vb));
    const bool two = rbk && rbv;
    const int n_loads = row1 > row0 ? (row1 - row0) * (two ? 2 : (rbk || rbv ? 1 : 0)) : 0;
    const unsigned char* qt = a.ws + wh->qt_off + (size_t)it.group * wh->qt_stride;
    const float* qhdr = reinterpret_cast<const float*>(qt);
    const uint2* bfrag = reinterpret_cast<const uint2*>(qt + kQtHeaderBytes);
    float qsum[NG];
#pragma unroll
    for (int u = 0; u < NG; ++u) qsum[u] = qhdr[Heads<G>::head(lane & 3, u)];
    const float qscale = qhdr[8];
    const uint32_t one = a.one;

    // issue state (lane 0 only): next row / side / stage to load
    int iss_row = row0, iss_stage = 0;
    bool iss_v = !rbk;
    const uint8_t* kbase = a.cache + koff;
    const uint8_t* vbase = a.cache + voff;
    auto issue_next = [&]() {
      const uint32_t bytes = iss_v ? rbv : rbk;
      const uint8_t* src = (iss_v ? vbase : kbase) +
                           row_offset(0, bytes, gr.seq, iss_row, a.page_table, a.pages_per_seq, a.rows_per_seq);
      const uint32_t bar = smem_addr(&bars[iss_stage]);
      mbar_arrive_expect_tx(bar, bytes);
      bulk_g2s(smem_addr(ring + (size_t)iss_stage * stage_bytes), src, bytes, bar);
      if (two && !iss_v) {
        iss_v = true;
      } else {
        iss_v = !rbk;
        ++iss_row;
      }
      if (++iss_stage == nstage) iss_stage = 0;
    };
    int issued = min(n_loads, nstage);
    if (lane == 0)
      for (int k = 0; k < issued; ++k) issue_next();
    outstanding = issued;

    // wait for the next stage; returns its buffer or nullptr on timeout
    auto acquire = [&]() -> const uint8_t* {
      const bool ok = __all_sync(
          0xffffffffu, mbar_wait_bounded(smem_addr(&bars[wait_stage]), (phase_bits >> wait_stage) & 1u, kWaitLimitNs));
      if (!ok) return nullptr;
      phase_bits ^= 1u << wait_stage;
      return ring + (size_t)wait_stage * stage_bytes;
    };
    // release the stage just consumed and refill it with the next load of this item
    auto release = [&]() {
      __syncwarp();
      --outstanding;
      if (++wait_stage == nstage) wait_stage = 0;
      if (issued < n_loads) {
        if (lane == 0) {
          fence_proxy_async_smem();
          issue_next();
        }
        ++issued;
        ++outstanding;
      }
    };

    for (int row = row0; row < row1; ++row) {
      float s[8][NG][2];
      // ---- K row ----
      if (rbk) {
        const uint8_t* buf = acquire();
        if (!buf) {
          failed = true;
          break;
        }
        k_row_dispatch<G>(kb, buf, kr, bfrag, qsum, qscale, one, s);
        release();
      } else {
#pragma unroll
        for (int t = 0; t < 8; ++t)
#pragma unroll
          for (int u = 0; u < NG; ++u) s[t][u][0] = s[t][u][1] = 0.f;
      }
      if ((row + 1) * kRowTokens > T) {  // only the last row of a sequence has masked tokens
        const int tbase = row * kRowTokens + (lane >> 2);
#pragma unroll
        for (int u = 0; u < NG; ++u)
#pragma unroll
          for (int t = 0; t < 8; ++t) {
            if (tbase + 16 * t >= T) s[t][u][0] = -INFINITY;
            if (tbase + 16 * t + 8 >= T) s[t][u][1] = -INFINITY;
          }
      }
      uint32_t bv[8][2];
      bool rescale = false;
      float alpha[NG];
      if (vc == 1)
        row_softmax<G, 1>(s, st, alpha, rescale, bv);
      else if (vc == 2)
        row_softmax<G, 2>(s, st, alpha, rescale, bv);
      else
        row_softmax<G, 0>(s, st, alpha, rescale, bv);
      // ---- V row ----
      if (rbv) {
        if (__any_sync(0xffffffffu, rescale)) {
          for (int mu = 0; mu < nmu; ++mu) {
            float* o = osm + (mu * 32 + lane) * NO;
#pragma unroll
            for (int k = 0; k < NO; ++k) o[k] *= alpha[NG == 2 ? (k & 1) : 0];
          }
        }
        const uint8_t* buf = acquire();
        if (!buf) {
          failed = true;
          break;
        }
        v_row_dispatch<G>(vb, buf, vr, bv, one, osm);
        release();
      }
    }
    if (failed) break;
    // ---- write the partial of this item ----
    __syncwarp();
#pragma unroll
    for (int u = 0; u < NG; ++u) {
      float l = st.l[u], c = st.c[u];
      l += __shfl_xor_sync(0xffffffffu, l, 4);
      l += __shfl_xor_sync(0xffffffffu, l, 8);
      l += __shfl_xor_sync(0xffffffffu, l, 16);
      c += __shfl_xor_sync(0xffffffffu, c, 4);
      c += __shfl_xor_sync(0xffffffffu, c, 8);
      c += __shfl_xor_sync(0xffffffffu, c, 16);
      if (vc == 0) c = l;
      const int g = Heads<G>::head(lane & 3, u);
      float* pg = part + g * gstride;
      if ((lane >> 2) == 0) {
        pg[0] = st.m[u];
        pg[1] = l;
      }
      for (int mu = 0; mu < nmu; ++mu) {
        const float* o = osm + (mu * 32 + lane) * NO;
        // G = 4: [ch0, ch1]; G = 8: [ch0 head 2j, ch0 head 2j+1, ch1 head 2j, ch1 head 2j+1]
        const float o0 = NO == 2 ? o[0] : o[u], o1 = NO == 2 ? o[1] : o[2 + u];
        const int ch0 = 16 * mu + (lane >> 2), ch1 = ch0 + 8;
        if (ch0 < vr) pg[4 + ch0] = (o0 - c) * vout;
        if (ch1 < vr) pg[4 + ch1] = (o1 - c) * vout;
      }
    }
    __syncwarp();
  }
  if (failed) {
    if (lane == 0) atomicOr(&g_status, 1u);
    // drain the copies still in flight before the shared memory goes away
    for (int k = 0; k < outstanding; ++k) {
      if (!mbar_wait_bounded(smem_addr(&bars[wait_stage]), (phase_bits >> wait_stage) & 1u, kWaitLimitNs)) break;
      phase_bits ^= 1u << wait_stage;
      if (++wait_stage == nstage) wait_stage = 0;
    }
  }
}

// ---------------------------------------------------------------------------------------
// a7: combine chunks + back-projection
//   per query head: m* = max over chunks, l* = sum 2^(m - m*) l, zbar = Delta_V (sum 2^(m - m*)
//   acc / l* - 2^{b-1} + 1/2), o = mu_V + W_V zbar (zeros for an empty sequence).
// ---------------------------------------------------------------------------------------
template <int G>
__global__ void __launch_bounds__(kHeadThreads) combine_kernel(DecodeArgs a) {
  constexpr int SPP = kVecPass / G;
  extern __shared__ __align__(16) float csm[];
  float* Ws = csm;                  // [kD][kD]     W_V row i = channel i
  float* Zs = Ws + kD * kD;         // [kD][kZLd]   zbar of this pass, [channel][vector]
  float* mus = Zs + kD * kZLd;      // [kD]         mu_V
  float* wts = mus + kD;            // [kVecPass][kWtChunk] normalised chunk weights
  __shared__ float vinfo_m[kVecPass], vinfo_inv_l[kVecPass];
  __shared__ int vinfo_first[kVecPass], vinfo_n[kVecPass], vinfo_g[kVecPass];
  const WsHeader* wh = reinterpret_cast<const WsHeader*>(a.ws);
  const WsGroup* groups = reinterpret_cast<const WsGroup*>(a.ws + wh->groups_off);
  const float* parts = reinterpret_cast<const float*>(a.ws + wh->part_off);
  const int S = wh->n_seqs;
  const int* hg = reinterpret_cast<const int*>(a.ws + wh->hg_off) + (size_t)blockIdx.x * S;
  const WsGroup g0 = groups[hg[0]];
  const HeadEntry hv = head_table(a.block)[g0.v_head];
  const float* pool = param_pool(a.block);
  const int rv = hv.r, layer = g0.layer, kv = g0.kv;
  const int tid = threadIdx.x;
  const float cen = rv > 0 ? (float)(1 << (hv.b - 1)) - 0.5f : 0.f;
  stage_basis(pool + hv.w_off, rv, kD, Ws);
  if (tid < kD) mus[tid] = pool[hv.mu_off + tid];
  for (int s0 = 0; s0 < S; s0 += SPP) {
    const int ns = min(SPP, S - s0), nv = ns * G;
    __syncthreads();  // basis staged; the previous pass is done with Zs
    // (1) per vector (warp w: vectors w, w + 8, w + 16, w + 24): m* = max over the chunks and
    //     l* = sum 2^(m - m*) l, lanes over chunks, merged online (a chunk with no tokens has
    //     m = -inf and no value entries; its weight is zero).  The four vectors' loads are
    //     issued together.
    const int warp = tid >> 5, lane = tid & 31;
    constexpr int NU = kVecPass / (kHeadThreads / 32);
    {
      const float* pg0[NU];
      int ni[NU];
      float M[NU], Lsum[NU];
      int kmax = 0;
#pragma unroll
      for (int u = 0; u < NU; ++u) {
        const int v = warp + 8 * u;
        const WsGroup gr = groups[hg[s0 + min(v, nv - 1) / G]];
        ni[u] = (v < nv && a.seq_lens[gr.seq] > 0) ? gr.n_items : 0;
        pg0[u] = parts + (size_t)gr.first_item * wh->part_stride + (v % G) * wh->g_stride;
        M[u] = -INFINITY;
        Lsum[u] = 0.f;
        kmax = max(kmax, ni[u]);
        if (v < nv && lane == 0) {
          vinfo_first[v] = ni[u] > 0 ? gr.first_item : -1;
          vinfo_n[v] = ni[u];
          vinfo_g[v] = v % G;
        }
      }
      for (int k = lane; k < kmax; k += 32) {
        float mk[NU], lk[NU];
#pragma unroll
        for (int u = 0; u < NU; ++u) {
          const bool ok = k < ni[u];
          mk[u] = ok ? pg0[u][(size_t)k * wh->part_stride] : -INFINITY;
          lk[u] = ok ? pg0[u][(size_t)k * wh->part_stride + 1] : 0.f;
        }
#pragma unroll
        for (int u = 0; u < NU; ++u) {
          if (mk[u] == -INFINITY) continue;
          const float mn = fmaxf(M[u], mk[u]);
          Lsum[u] = Lsum[u] * exp2f(M[u] - mn) + lk[u] * exp2f(mk[u] - mn);
          M[u] = mn;
        }
      }
#pragma unroll
      for (int u = 0; u < NU; ++u) {
#pragma unroll
        for (int o = 16; o; o >>= 1) {
          const float mo = __shfl_xor_sync(0xffffffffu, M[u], o), lo = __shfl_xor_sync(0xffffffffu, Lsum[u], o);
          const float mn = fmaxf(M[u], mo);
          if (mn != -INFINITY) {
            Lsum[u] = Lsum[u] * exp2f(M[u] - mn) + lo * exp2f(mo - mn);
            M[u] = mn;
          }
        }
        const int v = warp + 8 * u;
        if (v < nv && lane == 0) {
          vinfo_m[v] = M[u];
          vinfo_inv_l[v] = ni[u] > 0 ? 1.f / Lsum[u] : 0.f;
        }
      }
    }
    __syncthreads();
    // (2) zbar[v][i] = Delta (sum_k w_k acc_k[i] - 2^{b-1} + 1/2) with w_k = 2^(m_k - m*) / l*.
    //     Rounds of kWtChunk chunks: the weights of a round are computed one (vector, chunk) per
    //     thread into shared memory; then thread (channel i, vector parity) sums over them in
    //     blocks of 4 vectors x 8 chunks whose 32 loads are all issued before any is used.
    {
      const int i = tid & (kD - 1), par = tid >> 7;
      int kmax = 0;
      for (int v = 0; v < nv; ++v) kmax = max(kmax, vinfo_n[v]);
      float acc[kVecPass / 2];
#pragma unroll
      for (int q = 0; q < kVecPass / 2; ++q) acc[q] = 0.f;
      for (int k0 = 0; k0 < kmax; k0 += kWtChunk) {
        __syncthreads();  // the previous round's weights are consumed
        for (int idx = tid; idx < nv * kWtChunk; idx += kHeadThreads) {
          const int v = idx / kWtChunk, k = k0 + idx % kWtChunk;
          float w = 0.f;
          if (k < vinfo_n[v]) {
            const float mk = parts[(size_t)(vinfo_first[v] + k) * wh->part_stride + vinfo_g[v] * wh->g_stride];
            if (mk != -INFINITY) w = exp2f(mk - vinfo_m[v]) * vinfo_inv_l[v];
          }
          wts[idx] = w;
        }
        __syncthreads();
        if (i >= rv) continue;
        const int kr = min(kWtChunk, kmax - k0);
#pragma unroll
        for (int q0 = 0; q0 < kVecPass / 2; q0 += 4) {
          if (2 * q0 + par >= nv) break;
          for (int kb = 0; kb < kr; kb += 8) {
            float x[4][8];
#pragma unroll
            for (int qq = 0; qq < 4; ++qq) {
              const int v = 2 * (q0 + qq) + par;
              const int n = v < nv ? vinfo_n[v] - k0 : 0;
              const float* px = parts + (size_t)max(vinfo_first[v < nv ? v : 0], 0) * wh->part_stride +
                                (size_t)k0 * wh->part_stride + (v < nv ? vinfo_g[v] : 0) * wh->g_stride + 4 + i;
#pragma unroll
              for (int kk = 0; kk < 8; ++kk) x[qq][kk] = (kb + kk < n) ? px[(size_t)(kb + kk) * wh->part_stride] : 0.f;
            }
#pragma unroll
            for (int qq = 0; qq < 4; ++qq) {
              const int v = 2 * (q0 + qq) + par;
              if (v >= nv) break;
              const float* wv = wts + v * kWtChunk + kb;
#pragma unroll
              for (int kk = 0; kk < 8; ++kk) {
                const float w = (kb + kk < kWtChunk) ? wv[kk] : 0.f;
                acc[q0 + qq] += w != 0.f ? w * x[qq][kk] : 0.f;
              }
            }
          }
        }
      }
#pragma unroll
      for (int q = 0; q < kVecPass / 2; ++q) {
        const int v = 2 * q + par;
        if (v >= nv) break;
        Zs[i * kZLd + v] = (i < rv && vinfo_first[v] >= 0) ? hv.delta * (acc[q] - cen) : 0.f;
      }
    }
    __syncthreads();
    // thread: dims 4 (tid % 32) .. +3 for vectors 4 (tid / 32) .. +3
    const int d0 = 4 * (tid & 31), v0 = 4 * (tid >> 5);
    if (v0 < nv) {
      const float4 m4 = *reinterpret_cast<const float4*>(mus + d0);
      float4 o[4] = {m4, m4, m4, m4};
      for (int i = 0; i < rv; ++i) {
        const float4 w = *reinterpret_cast<const float4*>(Ws + i * kD + d0);
        const float4 z = *reinterpret_cast<const float4*>(Zs + i * kZLd + v0);
        const float zz[4] = {z.x, z.y, z.z, z.w};
#pragma unroll
        for (int v = 0; v < 4; ++v) {
          o[v].x += w.x * zz[v];
          o[v].y += w.y * zz[v];
          o[v].z += w.z * zz[v];
          o[v].w += w.w * zz[v];
        }
      }
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        const int vv = v0 + v;
        if (vv >= nv) break;
        const int seq = s0 + vv / G, g = vv % G;
        const bool empty = a.seq_lens[groups[hg[seq]].seq] <= 0;
        float* out = a.out + layer * a.o_sl + seq * a.o_ss + (long long)(kv * G + g) * kD + d0;
        const float4 y = empty ? make_float4(0.f, 0.f, 0.f, 0.f) : o[v];
        out[0] = y.x;  // the output is only 4-byte aligned in general
        out[1] = y.y;
        out[2] = y.z;
        out[3] = y.w;
      }
    }
  }
}

}  // namespace cobra
