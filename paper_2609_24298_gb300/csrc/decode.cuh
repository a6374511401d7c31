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
// a4: query projection
// ---------------------------------------------------------------------------------------
template <int G>
__global__ void __launch_bounds__(128) qproj_kernel(DecodeArgs a) {
  constexpr int NTK = Heads<G>::NTK;
  const WsHeader* wh = reinterpret_cast<const WsHeader*>(a.ws);
  const WsGroup gr = reinterpret_cast<const WsGroup*>(a.ws + wh->groups_off)[blockIdx.x];
  const HeadEntry hk = head_table(a.block)[gr.k_head];
  const float* pool = param_pool(a.block);
  unsigned char* qt = a.ws + wh->qt_off + (size_t)blockIdx.x * wh->qt_stride;
  const int r = hk.r;
  __shared__ float qs[G][kD];
  __shared__ float qv[G][kD];
  __shared__ float red[4];
  const int tid = threadIdx.x;
  const __nv_bfloat16* qp = a.q + gr.layer * a.q_sl + gr.seq * a.q_ss + (long long)gr.kv * G * kD;
#pragma unroll
  for (int g = 0; g < G; ++g) qv[g][tid] = __bfloat162float(qp[g * kD + tid]);
  __syncthreads();
  // q~[g][i] for channel i = tid
  const float scale = hk.delta * 0.088388347648318440f * 1.4426950408889634f;  // Delta/sqrt(128)*log2(e)
  float vals[G];
  float amax = 0.f;
#pragma unroll
  for (int g = 0; g < G; ++g) vals[g] = 0.f;
  if (tid < r) {
    const float* w = pool + hk.w_off + (size_t)tid * kD;
    for (int dd = 0; dd < kD; dd += 4) {
      const float4 wv = *reinterpret_cast<const float4*>(w + dd);
#pragma unroll
      for (int g = 0; g < G; ++g)
        vals[g] += wv.x * qv[g][dd] + wv.y * qv[g][dd + 1] + wv.z * qv[g][dd + 2] + wv.w * qv[g][dd + 3];
    }
#pragma unroll
    for (int g = 0; g < G; ++g) {
      vals[g] *= scale;
      amax = fmaxf(amax, fabsf(vals[g]));
    }
  }
  // power-of-two scale so that max |q~| lands in [256, 512)
#pragma unroll
  for (int o = 16; o; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
  if ((tid & 31) == 0) red[tid >> 5] = amax;
  __syncthreads();
  amax = fmaxf(fmaxf(red[0], red[1]), fmaxf(red[2], red[3]));
  int e = 0;
  if (amax > 0.f) {
    int ex;
    frexpf(amax, &ex);  // amax = m 2^ex, m in [0.5, 1)
    e = 9 - ex;
  }
  const float up = ldexpf(1.f, e);
#pragma unroll
  for (int g = 0; g < G; ++g) qs[g][tid] = vals[g] * up;
  __syncthreads();
  // sums of the fp16 hi+lo values actually fed to the MMA (scaled units)
  float* qhdr = reinterpret_cast<float*>(qt);
  if (tid < G) {
    float s = 0.f;
    for (int i = 0; i < r; ++i) {
      const float x = qs[tid][i];
      const __half h = __float2half_rn(x);
      const __half l = __float2half_rn(x - __half2float(h));
      s += __half2float(h) + __half2float(l);
    }
    qhdr[tid] = s;
  }
  if (tid == 0) qhdr[8] = ldexpf(1.f, -e);
  // B fragments [kappa][nt][lane] uint2: element (k, n) = hi or lo part of q~ of channel
  // 16 kappa + k for the query head of column n (see Heads)
  uint2* frag = reinterpret_cast<uint2*>(qt + kQtHeaderBytes);
  for (int idx = tid; idx < 8 * NTK * 32; idx += 128) {
    const int lane = idx & 31, nt = (idx >> 5) % NTK, kap = idx / (32 * NTK);
    const int j = lane & 3, n = lane >> 2;
    const int g = Heads<G>::col_head(nt, n), lo = Heads<G>::col_lo(nt, n);
    float e4[4];
    const int ks[4] = {2 * j, 2 * j + 1, 2 * j + 8, 2 * j + 9};
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int ch = 16 * kap + ks[u];
      float v = 0.f;
      if (ch < r) {
        const float x = qs[g][ch];
        const float h = __half2float(__float2half_rn(x));
        v = lo ? (x - h) : h;
      }
      e4[u] = v;
    }
    frag[(kap * 2 + nt) * 32 + lane] = make_uint2(pack_f16(e4[0], e4[1]), pack_f16(e4[2], e4[3]));
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

  for (int item = blockIdx.x * kDecodeWarps + warp; item < n_items && !failed; item += gridDim.x * kDecodeWarps) {
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
// ---------------------------------------------------------------------------------------
template <int G>
__global__ void __launch_bounds__(128) combine_kernel(DecodeArgs a) {
  const WsHeader* wh = reinterpret_cast<const WsHeader*>(a.ws);
  const WsGroup gr = reinterpret_cast<const WsGroup*>(a.ws + wh->groups_off)[blockIdx.x];
  const HeadEntry hv = head_table(a.block)[gr.v_head];
  const float* pool = param_pool(a.block);
  const float* parts = reinterpret_cast<const float*>(a.ws + wh->part_off);
  const int tid = threadIdx.x;
  float* out = a.out + gr.layer * a.o_sl + gr.seq * a.o_ss + (long long)gr.kv * G * kD;
  const int T = a.seq_lens[gr.seq];
  if (T <= 0) {
#pragma unroll
    for (int g = 0; g < G; ++g) out[g * kD + tid] = 0.f;
    return;
  }
  __shared__ float zbar[G][kD];
  __shared__ float wts[G][64];
  const int rv = hv.r, ni = gr.n_items;
  const float cen = hv.r > 0 ? (float)(1 << (hv.b - 1)) - 0.5f : 0.f;
  for (int g = 0; g < G; ++g) {
    float mstar = -INFINITY;
    for (int k = 0; k < ni; ++k) mstar = fmaxf(mstar, parts[(size_t)(gr.first_item + k) * wh->part_stride + g * wh->g_stride]);
    float lstar = 0.f, acc = 0.f;
    for (int k = 0; k < ni; ++k) {
      const float* pg = parts + (size_t)(gr.first_item + k) * wh->part_stride + g * wh->g_stride;
      const float w = (pg[0] == -INFINITY) ? 0.f : exp2f(pg[0] - mstar);
      lstar += w * pg[1];
      if (tid < rv && w != 0.f) acc += w * pg[4 + tid];
    }
    if (tid < rv) zbar[g][tid] = hv.delta * (acc / lstar - cen);
  }
  (void)wts;
  __syncthreads();
  const float* W = pool + hv.w_off;
  const float mu = pool[hv.mu_off + tid];
  float o[G];
#pragma unroll
  for (int g = 0; g < G; ++g) o[g] = mu;
  for (int i = 0; i < rv; ++i) {
    const float w = W[(size_t)i * kD + tid];
#pragma unroll
    for (int g = 0; g < G; ++g) o[g] += w * zbar[g][i];
  }
#pragma unroll
  for (int g = 0; g < G; ++g) out[g * kD + tid] = o[g];
}

}  // namespace cobra
