// Decode attention over the packed cache, in rank space (Table alg:kvrobin step 8; App. G).
//
// Three kernels per call:
//   qproj_kernel    q~_g = (Delta_K / sqrt d) log2(e) W_K^T q_g for the G query heads of a
//                   kv head, split into fp16 hi + lo, laid out as MMA B fragments.
//   decode_kernel   persistent warps over work items (token chunks of one (seq, layer, kv-head)).
//                   Each warp streams its chunk's K and V code rows into a private shared-
//                   memory ring with bulk async copies, unpacks codes in registers and runs
//                   f16 mma.sync with fp32 accumulation:
//                     scores  S[t][(g,hi|lo)] = sum_i code^K[t][i] q~[i][(g,hi|lo)]   (M = tokens)
//                     values  O[i][(g,hi|lo)] += sum_t code^V[t][i] P[t][(g,hi|lo)]  (M = channels)
//                   with an online softmax in base 2 between them.  Writes per-chunk
//                   partials (m, l, sum_t p_t c^V_t).
//   combine_kernel  merges the chunks of each (seq, layer, kv-head), dequantises the rank-space
//                   average and back-projects once: o = mu_V + W_V Delta_V (acc/l - 2^{b-1} + 1/2).
#pragma once

#include "common.cuh"

namespace cobra {

constexpr int kDecodeWarps = 4;
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
  int stage_bytes, nstage;
};

// ---------------------------------------------------------------------------------------
// a4: query projection
// ---------------------------------------------------------------------------------------
template <int G>
__global__ void __launch_bounds__(128) qproj_kernel(DecodeArgs a) {
  constexpr int NT = G / 4;
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
  if (tid < r) {
    const float* w = pool + hk.w_off + (size_t)tid * kD;
#pragma unroll
    for (int g = 0; g < G; ++g) vals[g] = 0.f;
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
  } else {
#pragma unroll
    for (int g = 0; g < G; ++g) vals[g] = 0.f;
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
  // B fragments: [kappa][nt][lane] uint2; element (k, n): channel 16 kappa + k, column n =
  // 2 (g mod 4) + (hi|lo) of query head g = 4 nt + n / 2.
  uint2* frag = reinterpret_cast<uint2*>(qt + kQtHeaderBytes);
  for (int idx = tid; idx < 8 * NT * 32; idx += 128) {
    const int lane = idx & 31, nt = (idx >> 5) % NT, kap = idx / (32 * NT);
    const int j = lane & 3, n = lane >> 2;
    const int g = 4 * nt + (n >> 1), lo = n & 1;
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
// ---------------------------------------------------------------------------------------
template <int G>
struct WarpState {
  static constexpr int NT = G / 4;
  float m[NT], l[NT], c[NT];
  float o[NT][8][4];
};

// K side: scores of one code row for the lane's query heads.  Returns scores in s[8][NT][2]
// (token t0 = 16 tau + lane/4 in [..][..][0], t1 = t0 + 8 in [..][..][1]), log2 units.
template <int G, int B>
__device__ __forceinline__ void k_row_scores(const uint8_t* stage, int rk, const uint2* bfrag, const float* qsum,
                                             float qscale, float (&s)[8][G / 4][2]) {
  constexpr int NT = G / 4;
  const int lane = threadIdx.x & 31;
  float acc[8][NT][4];
#pragma unroll
  for (int t = 0; t < 8; ++t)
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) acc[t][nt][0] = acc[t][nt][1] = acc[t][nt][2] = acc[t][nt][3] = 0.f;
  const int P = rk >> 1;
  const int nk = (P + 7) >> 3;
#pragma unroll
  for (int kap = 0; kap < 8; ++kap) {
    if (kap < nk) {
      const int sA = 8 * kap + (lane & 3), sB = sA + 4, pc = lane >> 2;
      uint32_t pa[16], pb[16];
      if (sA < P) {
        uint32_t w[B];
        load_piece<B>(stage + sA * 32 * B + pc * 4 * B, w);
        unpack_piece<B>(w, pa);
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) pa[i] = 0u;
      }
      if (sB < P) {
        uint32_t w[B];
        load_piece<B>(stage + sB * 32 * B + pc * 4 * B, w);
        unpack_piece<B>(w, pb);
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) pb[i] = 0u;
      }
      uint2 bf[NT];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) bf[nt] = bfrag[(kap * 2 + nt) * 32 + lane];
#pragma unroll
      for (int t = 0; t < 8; ++t)
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
          mma_f16(acc[t][nt], pa[2 * t], pa[2 * t + 1], pb[2 * t], pb[2 * t + 1], bf[nt].x, bf[nt].y);
    }
  }
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    const float qg = qsum[4 * nt + (lane & 3)];
#pragma unroll
    for (int t = 0; t < 8; ++t) {
      s[t][nt][0] = (acc[t][nt][0] + acc[t][nt][1] - Window<B>::off(2 * t) * qg) * qscale;
      s[t][nt][1] = (acc[t][nt][2] + acc[t][nt][3] - Window<B>::off(2 * t + 1) * qg) * qscale;
    }
  }
}

// V side: accumulate one code row into o (rank space) and the offset correction into c.
template <int G, int B>
__device__ __forceinline__ void v_row_accumulate(const uint8_t* stage, int rv, const uint32_t (&bv)[8][G / 4][2],
                                                 const float (&p)[8][G / 4][2], WarpState<G>& st) {
  constexpr int NT = G / 4;
  const int lane = threadIdx.x & 31;
  const int P = rv >> 1;
  const int nmu = (P + 7) >> 3;
#pragma unroll
  for (int mu = 0; mu < 8; ++mu) {
    if (mu < nmu) {
      const int sA = 8 * mu + (lane >> 3), sB = sA + 4, pc = lane & 7;
      uint32_t pa[16], pb[16];
      if (sA < P) {
        uint32_t w[B];
        load_piece<B>(stage + sA * 32 * B + pc * 4 * B, w);
        unpack_piece<B>(w, pa);
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) pa[i] = 0u;
      }
      if (sB < P) {
        uint32_t w[B];
        load_piece<B>(stage + sB * 32 * B + pc * 4 * B, w);
        unpack_piece<B>(w, pb);
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) pb[i] = 0u;
      }
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        float d[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int t = 0; t < 8; ++t) mma_f16(d, pa[2 * t], pb[2 * t], pa[2 * t + 1], pb[2 * t + 1], bv[t][nt][0], bv[t][nt][1]);
        st.o[nt][mu][0] += d[0];
        st.o[nt][mu][1] += d[1];
        st.o[nt][mu][2] += d[2];
        st.o[nt][mu][3] += d[3];
      }
    }
  }
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    float c = 0.f;
#pragma unroll
    for (int t = 0; t < 8; ++t) c += p[t][nt][0] * Window<B>::off(2 * t) + p[t][nt][1] * Window<B>::off(2 * t + 1);
    st.c[nt] += c;
  }
}

template <int G>
__device__ __forceinline__ void k_row_dispatch(int b, const uint8_t* stage, int rk, const uint2* bfrag, const float* qsum,
                                               float qscale, float (&s)[8][G / 4][2]) {
  switch (b) {
    case 1: k_row_scores<G, 1>(stage, rk, bfrag, qsum, qscale, s); break;
    case 2: k_row_scores<G, 2>(stage, rk, bfrag, qsum, qscale, s); break;
    case 3: k_row_scores<G, 3>(stage, rk, bfrag, qsum, qscale, s); break;
    case 4: k_row_scores<G, 4>(stage, rk, bfrag, qsum, qscale, s); break;
    case 5: k_row_scores<G, 5>(stage, rk, bfrag, qsum, qscale, s); break;
    case 6: k_row_scores<G, 6>(stage, rk, bfrag, qsum, qscale, s); break;
    case 7: k_row_scores<G, 7>(stage, rk, bfrag, qsum, qscale, s); break;
    default: k_row_scores<G, 8>(stage, rk, bfrag, qsum, qscale, s); break;
  }
}

template <int G>
__device__ __forceinline__ void v_row_dispatch(int b, const uint8_t* stage, int rv, const uint32_t (&bv)[8][G / 4][2],
                                               const float (&p)[8][G / 4][2], WarpState<G>& st) {
  switch (b) {
    case 1: v_row_accumulate<G, 1>(stage, rv, bv, p, st); break;
    case 2: v_row_accumulate<G, 2>(stage, rv, bv, p, st); break;
    case 3: v_row_accumulate<G, 3>(stage, rv, bv, p, st); break;
    case 4: v_row_accumulate<G, 4>(stage, rv, bv, p, st); break;
    case 5: v_row_accumulate<G, 5>(stage, rv, bv, p, st); break;
    case 6: v_row_accumulate<G, 6>(stage, rv, bv, p, st); break;
    case 7: v_row_accumulate<G, 7>(stage, rv, bv, p, st); break;
    default: v_row_accumulate<G, 8>(stage, rv, bv, p, st); break;
  }
}

template <int G>
__global__ void __launch_bounds__(kDecodeWarps * 32) decode_kernel(DecodeArgs a) {
  constexpr int NT = G / 4;
  extern __shared__ __align__(128) uint8_t smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nstage = a.nstage, stage_bytes = a.stage_bytes;
  uint8_t* ring = smem + (size_t)warp * nstage * stage_bytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + (size_t)kDecodeWarps * nstage * stage_bytes) + warp * nstage;
  if (lane == 0) {
    for (int i = 0; i < nstage; ++i) mbar_init(smem_addr(&bars[i]), 1);
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
  uint32_t phase_bits = 0;  // parity of the next wait per stage
  bool failed = false;
  int outstanding = 0;      // loads issued but not yet waited for (stages are used in order)
  int next_wait_stage = 0;

  for (int item = blockIdx.x * kDecodeWarps + warp; item < n_items && !failed; item += gridDim.x * kDecodeWarps) {
    const WsItem it = items[item];
    const WsGroup gr = groups[it.group];
    const HeadEntry hk = heads[gr.k_head], hv = heads[gr.v_head];
    const int T = a.seq_lens[gr.seq];
    const int rows_valid = (T + kRowTokens - 1) / kRowTokens;
    const int row0 = it.row_begin, row1 = min(it.row_end, rows_valid);
    float* part = parts + (size_t)item * pstride;
    WarpState<G> st;
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      st.m[nt] = -INFINITY;
      st.l[nt] = 0.f;
      st.c[nt] = 0.f;
#pragma unroll
      for (int mu = 0; mu < 8; ++mu) st.o[nt][mu][0] = st.o[nt][mu][1] = st.o[nt][mu][2] = st.o[nt][mu][3] = 0.f;
    }
    const uint32_t rbk = hk.r > 0 ? 16u * hk.r * hk.b : 0u, rbv = hv.r > 0 ? 16u * hv.r * hv.b : 0u;
    if (rbk > (uint32_t)stage_bytes || rbv > (uint32_t)stage_bytes) {
      // a row that does not fit the staging buffer is never copied; report and leave an
      // empty chunk (m = -inf, l = 0)
      if (lane == 0) atomicOr(&g_status, 2u);
      if (lane < G) {
        part[lane * gstride + 0] = -INFINITY;
        part[lane * gstride + 1] = 0.f;
      }
      continue;
    }
    const int loads_per_row = (rbk ? 1 : 0) + (rbv ? 1 : 0);
    const int n_loads = row1 > row0 ? (row1 - row0) * loads_per_row : 0;
    const unsigned char* qt = a.ws + wh->qt_off + (size_t)it.group * wh->qt_stride;
    const float* qhdr = reinterpret_cast<const float*>(qt);
    const uint2* bfrag = reinterpret_cast<const uint2*>(qt + kQtHeaderBytes);
    float qsum[G];
#pragma unroll
    for (int g = 0; g < G; ++g) qsum[g] = qhdr[g];
    const float qscale = qhdr[8];

    // load n of this item -> (row, side)
    auto load_src = [&](int n, uint32_t& bytes) -> const uint8_t* {
      const int row = row0 + n / loads_per_row;
      const bool is_v = (loads_per_row == 2) ? (n & 1) : (rbk == 0);
      const HeadEntry& h = is_v ? hv : hk;
      bytes = is_v ? rbv : rbk;
      return a.cache + row_offset(h.cache_off, bytes, gr.seq, row, a.page_table, a.pages_per_seq, a.rows_per_seq);
    };
    // prologue: fill the ring
    int issued = 0;
    if (lane == 0) {
      for (; issued < n_loads && issued < nstage; ++issued) {
        const int stg = (next_wait_stage + issued) % nstage;
        uint32_t bytes;
        const uint8_t* src = load_src(issued, bytes);
        const uint32_t bar = smem_addr(&bars[stg]);
        mbar_arrive_expect_tx(bar, bytes);
        bulk_g2s(smem_addr(ring + (size_t)stg * stage_bytes), src, bytes, bar);
      }
    }
    issued = __shfl_sync(0xffffffffu, issued, 0);
    outstanding = issued;

    int consumed = 0;
    for (int row = row0; row < row1; ++row) {
      float s[8][NT][2];
      // ---- K row ----
      if (rbk) {
        const int stg = next_wait_stage;
        const bool ok = __all_sync(0xffffffffu, mbar_wait_bounded(smem_addr(&bars[stg]), (phase_bits >> stg) & 1u, kWaitLimitNs));
        if (!ok) {
          failed = true;
          break;
        }
        phase_bits ^= 1u << stg;
        k_row_dispatch<G>(hk.b, ring + (size_t)stg * stage_bytes, hk.r, bfrag, qsum, qscale, s);
        __syncwarp();
        ++consumed;
        --outstanding;
        next_wait_stage = (next_wait_stage + 1) % nstage;
        if (lane == 0 && issued < n_loads) {
          fence_proxy_async_smem();
          uint32_t bytes;
          const uint8_t* src = load_src(issued, bytes);
          const uint32_t bar = smem_addr(&bars[stg]);
          mbar_arrive_expect_tx(bar, bytes);
          bulk_g2s(smem_addr(ring + (size_t)stg * stage_bytes), src, bytes, bar);
        }
        if (issued < n_loads) {
          ++issued;
          ++outstanding;
        }
      } else {
#pragma unroll
        for (int t = 0; t < 8; ++t)
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) s[t][nt][0] = s[t][nt][1] = 0.f;
      }
      // ---- online softmax (base 2) ----
      const int tbase = row * kRowTokens + (lane >> 2);
      float p[8][NT][2];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        float mx = -INFINITY;
#pragma unroll
        for (int t = 0; t < 8; ++t) {
          if (tbase + 16 * t >= T) s[t][nt][0] = -INFINITY;
          if (tbase + 16 * t + 8 >= T) s[t][nt][1] = -INFINITY;
          mx = fmaxf(mx, fmaxf(s[t][nt][0], s[t][nt][1]));
        }
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
        const float mnew = fmaxf(st.m[nt], mx);
        const float alpha = exp2f(st.m[nt] - mnew);
        st.m[nt] = mnew;
        st.l[nt] *= alpha;
        st.c[nt] *= alpha;
#pragma unroll
        for (int mu = 0; mu < 8; ++mu) {
          st.o[nt][mu][0] *= alpha;
          st.o[nt][mu][1] *= alpha;
          st.o[nt][mu][2] *= alpha;
          st.o[nt][mu][3] *= alpha;
        }
        float ls = 0.f;
#pragma unroll
        for (int t = 0; t < 8; ++t) {
          p[t][nt][0] = exp2f(s[t][nt][0] - mnew);
          p[t][nt][1] = exp2f(s[t][nt][1] - mnew);
          ls += p[t][nt][0] + p[t][nt][1];
        }
        st.l[nt] += ls;
      }
      // ---- V row ----
      if (rbv) {
        uint32_t bv[8][NT][2];
#pragma unroll
        for (int t = 0; t < 8; ++t)
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            const float h0 = __half2float(__float2half_rn(p[t][nt][0]));
            const float h1 = __half2float(__float2half_rn(p[t][nt][1]));
            bv[t][nt][0] = movmatrix_t(pack_f16(h0, p[t][nt][0] - h0));
            bv[t][nt][1] = movmatrix_t(pack_f16(h1, p[t][nt][1] - h1));
          }
        const int stg = next_wait_stage;
        const bool ok = __all_sync(0xffffffffu, mbar_wait_bounded(smem_addr(&bars[stg]), (phase_bits >> stg) & 1u, kWaitLimitNs));
        if (!ok) {
          failed = true;
          break;
        }
        phase_bits ^= 1u << stg;
        v_row_dispatch<G>(hv.b, ring + (size_t)stg * stage_bytes, hv.r, bv, p, st);
        __syncwarp();
        ++consumed;
        --outstanding;
        next_wait_stage = (next_wait_stage + 1) % nstage;
        if (lane == 0 && issued < n_loads) {
          fence_proxy_async_smem();
          uint32_t bytes;
          const uint8_t* src = load_src(issued, bytes);
          const uint32_t bar = smem_addr(&bars[stg]);
          mbar_arrive_expect_tx(bar, bytes);
          bulk_g2s(smem_addr(ring + (size_t)stg * stage_bytes), src, bytes, bar);
        }
        if (issued < n_loads) {
          ++issued;
          ++outstanding;
        }
      }
    }
    if (failed) break;
    // ---- write the partial of this item ----
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      float l = st.l[nt], c = st.c[nt];
      l += __shfl_xor_sync(0xffffffffu, l, 4);
      l += __shfl_xor_sync(0xffffffffu, l, 8);
      l += __shfl_xor_sync(0xffffffffu, l, 16);
      c += __shfl_xor_sync(0xffffffffu, c, 4);
      c += __shfl_xor_sync(0xffffffffu, c, 8);
      c += __shfl_xor_sync(0xffffffffu, c, 16);
      const int g = 4 * nt + (lane & 3);
      float* pg = part + g * gstride;
      if ((lane >> 2) == 0) {
        pg[0] = st.m[nt];
        pg[1] = l;
      }
      const int rv = hv.r;
#pragma unroll
      for (int mu = 0; mu < 8; ++mu) {
        const int ch0 = 16 * mu + (lane >> 2), ch1 = ch0 + 8;
        if (ch0 < rv) pg[4 + ch0] = (st.o[nt][mu][0] + st.o[nt][mu][1]) - c;
        if (ch1 < rv) pg[4 + ch1] = (st.o[nt][mu][2] + st.o[nt][mu][3]) - c;
      }
    }
  }
  if (failed) {
    if (lane == 0) atomicOr(&g_status, 1u);
    // drain the copies still in flight before the shared memory goes away
    for (int k = 0; k < outstanding; ++k) {
      const int stg = (next_wait_stage + k) % nstage;
      if (!mbar_wait_bounded(smem_addr(&bars[stg]), (phase_bits >> stg) & 1u, kWaitLimitNs)) break;
      phase_bits ^= 1u << stg;
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
