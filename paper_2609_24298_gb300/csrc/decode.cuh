// Decode attention over the packed cache, in rank space (Table alg:kvrobin step 8; App. G).
//
// Three kernels per call (the first and last in decode_heads.cuh):
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
// a5 + a6: chunked rank-space scan
//
// Per warp and work item (a run of code rows of one (seq, layer, kv head)):
//  * each stage of the warp's shared-memory ring holds one K row and the V row of the same
//    tokens, both copied with cp.async.bulk onto one mbarrier; the copies are issued by one
//    lane under a predicate, so the warp never diverges;
//  * scores s_t (log2 units) come from the K codes by f16 MMA; probabilities are taken
//    against a reference max that is raised (and the accumulators rescaled) only when a
//    row's max exceeds it by more than kTau, so most rows need no rescale;
//  * the V MMA accumulates O[i] = sum_t f_t A_t[i] over the fed probabilities f_t.  Two
//    constant rows appended after the last channel give, in the same accumulators, the sum
//    of the fed values c (row r: A = 1) and the normaliser l (row r + 1: A = 2^(k - kmin),
//    which undoes each register's window), so both are rescaled with O.
// Loops over k-tiles (K side) and channel tiles (V side) stay rolled to keep each bit width's
// code small; the 8 token tiles of a row are unrolled.
// ---------------------------------------------------------------------------------------
constexpr float kTau = 8.f;    // fed probabilities stay below 2^kTau (fp16 range)
constexpr int kMaxVTiles = 9;  // channel tiles of the V accumulators: 8 + the one holding rows r, r+1

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
  const int nk = ((rk >> 1) + 7) >> 3;
  // lane's pieces: strips 8 kappa + (lane & 3) and + 4, piece lane >> 2.  A partial last
  // k-tile reads past the row (at most 7 strips, still inside the warp's shared memory): any
  // word bits unpack to finite values, and channels past r multiply q~ = 0.
  const uint8_t* pa = stage + (lane & 3) * 32 * B + (lane >> 2) * 4 * B;
  const uint2* bq = bfrag + lane;
#pragma unroll 1
  for (int kap = 0; kap < nk; ++kap) {
    uint32_t wa[B], wb[B];
    load_piece<B>(pa, wa);
    load_piece<B>(pa + 4 * 32 * B, wb);
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
    bq += NTK * 32;
  }
  // acc = Qsum + 2^(k-10) * sum_i q~_i code_i, Qsum = sum of the q~ fed to the MMA.  b >= 3
  // uses one window for every register, so Qsum shifts every token's score alike and softmax
  // ignores it; b = 1, 2 mix windows, so Qsum is removed before the per-token rescale:
  // s = acc * sc - Qsum * sc with sc = scale 2^(10-k).
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
        s[t][u][0] = fmaf(v0, sc0, -qsum[u] * sc0);
        s[t][u][1] = fmaf(v1, sc1, -qsum[u] * sc1);
      } else {
        s[t][u][0] = v0 * sc0;
        s[t][u][1] = v1 * sc1;
      }
    }
  }
}

// f16x2 constant of the normaliser row for register rho: 2^(k(rho) - kmin) in both halves
template <int B>
__host__ __device__ constexpr uint32_t unshift_h2(int rho) {
  return (((uint32_t)(Window<B>::k(rho) - Window<B>::kmin() + 15) << 10) * 0x00010001u);
}

// V side: add one code row's rank-space contribution into the shared-memory accumulators.
// The tile holding strip P = r/2 is always processed: its lanes on strip P feed the constant
// rows r (code 0, i.e. 1.0: zero words) and r + 1 (the per-register window factor).
template <int G, int B>
__device__ __forceinline__ void v_row_accumulate(const uint8_t* stage, int rv, const uint32_t (&bv)[8][2],
                                                 uint32_t one, float* osm) {
  constexpr int NO = OAcc<G>::N;
  const int lane = threadIdx.x & 31;
  const int P = rv >> 1;
  const int nfull = P >> 3;
  // lane's pieces: strips 8 mu + (lane >> 3) and + 4, piece lane & 7
  const uint8_t* pa = stage + (lane >> 3) * 32 * B + (lane & 7) * 4 * B;
  float* o = osm + lane * NO;
  auto tile = [&](bool check, int mu) {
    uint32_t wa[B], wb[B];
    bool la = false, lb = false;  // this lane feeds the normaliser row (strip P, odd channel)
    if (check) {
      const int sA = 8 * mu + (lane >> 3);
      load_piece_or_zero<B>(pa, sA < P, wa);
      load_piece_or_zero<B>(pa + 4 * 32 * B, sA + 4 < P, wb);
      la = B <= 2 && sA == P && (lane & 4);
      lb = B <= 2 && sA + 4 == P && (lane & 4);
    } else {
      load_piece<B>(pa, wa);
      load_piece<B>(pa + 4 * 32 * B, wb);
    }
    // fresh accumulators per row: the running sums in shared memory are dominated by the unit
    // code offsets, so they are only ever updated with round-to-nearest fp32 adds
    float d[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
    for (int t = 0; t < 8; ++t) {
      uint32_t a0 = unpack_reg<B>(wa, 2 * t, one), a1 = unpack_reg<B>(wb, 2 * t, one);
      uint32_t a2 = unpack_reg<B>(wa, 2 * t + 1, one), a3 = unpack_reg<B>(wb, 2 * t + 1, one);
      if constexpr (B <= 2) {
        if (check) {
          a0 = la ? unshift_h2<B>(2 * t) : a0;
          a2 = la ? unshift_h2<B>(2 * t + 1) : a2;
          a1 = lb ? unshift_h2<B>(2 * t) : a1;
          a3 = lb ? unshift_h2<B>(2 * t + 1) : a3;
        }
      }
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
  tile(true, nfull);
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

// b = 0 stands for a head with r_V = 0: only the constant rows (one window class)
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
    case 8: v_row_accumulate<G, 8>(stage, rv, bv, one, osm); break;
    default: v_row_accumulate<G, 3>(stage, 0, bv, one, osm); break;
  }
}

template <int G>
__host__ __device__ constexpr size_t decode_osm_bytes() {
  return (size_t)kMaxVTiles * 32 * OAcc<G>::N * sizeof(float);
}
// the group's q~ MMA B fragments, copied into the warp's shared memory once per work item
template <int G>
__host__ __device__ constexpr uint32_t decode_qfrag_bytes() {
  return 8u * Heads<G>::NTK * 32u * 8u;
}

// VC is the V bit width's window class: 0 = one window for every register (b >= 3, or no V
// codes), 1 or 2 = the b = 1 / b = 2 windows.  V codes read 1 + code * 2^(k-10) with a
// per-register window k, so each token's probability is fed to the MMA pre-scaled by
// 2^(kmin - k) (folded into the exponent): the products then carry the single scale
// 2^(kmin-10), and the unit offsets add up to the plain sum of the fed values.
template <int VC>
struct VWin {
  static constexpr int B = VC == 0 ? 3 : VC;
  __device__ static constexpr float shift(int rho) {  // kmin - k (<= 0)
    return VC == 0 ? 0.f : (float)(Window<B>::kmin() - Window<B>::k(rho));
  }
};

// Probabilities of one row against the reference max, as the V side's MMA B operands: the
// 16 x 8 probability tile of token tile t in C-fragment layout (row t0 or t1, columns 2j,
// 2j+1), transposed by movmatrix.  Each fed value is rounded to fp16 once; the same value
// enters O, c and l through the MMA, so the weights stay exactly normalised.
template <int G, int VC>
__device__ __forceinline__ void row_probs(const float (&s)[8][G / 4][2], const float (&mref)[G / 4],
                                          uint32_t (&bv)[8][2]) {
  constexpr int NG = G / 4;
  float pf[8][NG][2];
#pragma unroll
  for (int u = 0; u < NG; ++u)
#pragma unroll
    for (int t = 0; t < 8; ++t) {
      pf[t][u][0] = ex2_approx(s[t][u][0] + (VWin<VC>::shift(2 * t) - mref[u]));
      pf[t][u][1] = ex2_approx(s[t][u][1] + (VWin<VC>::shift(2 * t + 1) - mref[u]));
    }
#pragma unroll
  for (int t = 0; t < 8; ++t) {
    const float c0 = pf[t][0][0], c1 = NG == 2 ? pf[t][NG - 1][0] : 0.f;
    const float c2 = pf[t][0][1], c3 = NG == 2 ? pf[t][NG - 1][1] : 0.f;
    bv[t][0] = movmatrix_t(pack_f16(c0, c1));
    bv[t][1] = movmatrix_t(pack_f16(c2, c3));
  }
}

// Per-warp state of the scan that outlives a work item.
struct ScanWarp {
  uint8_t* ring;
  float* osm;
  uint2* qfrag;
  uint64_t* bars;
  int ring_bytes, lane;
  bool leader, failed;
  uint32_t phase_bits;  // parity of the next wait per barrier
  int wait_stage, nstage, outstanding;
};

// One work item.  BK / BV > 0 fix the K / V bit widths at compile time (the common widths
// get their own copy of the row loop); 0 dispatches on the runtime widths row by row.
template <int G, int BK, int BV>
__device__ __forceinline__ void scan_item(const DecodeArgs& a, ScanWarp& w, int item) {
  constexpr int NG = G / 4, NO = OAcc<G>::N;
  const int lane = w.lane;
  const bool leader = w.leader;
  const WsHeader* wh = reinterpret_cast<const WsHeader*>(a.ws);
  const WsGroup* groups = reinterpret_cast<const WsGroup*>(a.ws + wh->groups_off);
  const WsItem* items = reinterpret_cast<const WsItem*>(a.ws + wh->items_off);
  const HeadEntry* heads = head_table(a.block);
  float* parts = reinterpret_cast<float*>(a.ws + wh->part_off);
  const int gstride = wh->g_stride, pstride = wh->part_stride;
  const WsItem it = items[item];
  const WsGroup gr = groups[it.group];
  const int kr = heads[gr.k_head].r, vr = heads[gr.v_head].r;
  const int kb = BK > 0 ? BK : heads[gr.k_head].b, vb = BV > 0 ? BV : heads[gr.v_head].b;
  const uint64_t koff = heads[gr.k_head].cache_off, voff = heads[gr.v_head].cache_off;
  const int T = a.seq_lens[gr.seq];
  const int rows_valid = (T + kRowTokens - 1) / kRowTokens;
  const int row0 = it.row_begin, row1 = min(it.row_end, rows_valid);
  float* part = parts + (size_t)it.slot * pstride;
  const uint32_t rbk = kr > 0 ? 16u * kr * kb : 0u, rbv = vr > 0 ? 16u * vr * vb : 0u;
  // one stage = this item's K row + V row (every load of the previous item has been
  // consumed, so the whole ring is free)
  const uint32_t kst = (rbk + 127u) & ~127u;
  const int stage_bytes = (int)max(kst + ((rbv + 127u) & ~127u), 128u);
  w.nstage = min(kMaxStages, w.ring_bytes / stage_bytes);
  w.wait_stage = 0;
  if (w.nstage < 1) {
    // a row pair that does not fit the staging ring is never copied; report and leave an
    // empty chunk (m = -inf, l = 0)
    if (leader) atomicOr(&g_status, 2u);
    if (lane < G) {
      part[lane * gstride + 0] = -INFINITY;
      part[lane * gstride + 1] = 0.f;
    }
    return;
  }
  float* osm = w.osm;
  float mref[NG];
#pragma unroll
  for (int u = 0; u < NG; ++u) mref[u] = -INFINITY;
  const int ntile = (vr >> 4) + 1;  // V accumulator tiles incl. the constant rows
  for (int k = 0; k < ntile * NO; ++k) osm[k * 32 + lane] = 0.f;
  // V window class (see VWin) and the factor 2^(10 - kmin) that turns the fed products back
  // into codes
  const int vc = (vr > 0 && vb <= 2) ? vb : 0;
  const int vbd = vr > 0 ? vb : 0;
  const float vout = vr == 0 ? 0.f : (float)(1 << (vb == 1 ? 5 : vb == 2 ? 6 : vb));
  const int n_loads = (row1 > row0 && (rbk || rbv)) ? row1 - row0 : 0;
  const unsigned char* qt = a.ws + wh->qt_off + (size_t)it.group * wh->qt_stride;
  const float* qhdr = reinterpret_cast<const float*>(qt);
  const uint2* bfrag = w.qfrag;  // filled together with the item's first stage
  float qsum[NG];
#pragma unroll
  for (int u = 0; u < NG; ++u) qsum[u] = qhdr[Heads<G>::head(lane & 3, u)];
  const float qscale = qhdr[8];
  const uint32_t one = a.one;

  // issue state: next row and stage to load (every lane tracks it; lane 0 issues).  In a
  // contiguous cache the item's rows follow one another, so the sources advance by a row;
  // a paged cache looks each row's page up.
  int iss_row = row0, iss_stage = 0;
  const uint8_t* kbase = a.cache + koff;
  const uint8_t* vbase = a.cache + voff;
  const int* const page_table = a.page_table;
  const int pages_per_seq = a.pages_per_seq, seq = gr.seq;
  const size_t slot0 = (size_t)seq * a.rows_per_seq + row0;
  const uint8_t* ksrc = kbase + slot0 * rbk;
  const uint8_t* vsrc = vbase + slot0 * rbv;
  const uint32_t ring0 = smem_addr(w.ring), bar0 = smem_addr(w.bars);
  const int nstage = w.nstage;
  auto issue_next = [&]() {
    const uint8_t* ks = ksrc;
    const uint8_t* vs = vsrc;
    if (page_table) {
      ks = kbase + row_offset(0, rbk, seq, iss_row, page_table, pages_per_seq, 0);
      vs = vbase + row_offset(0, rbv, seq, iss_row, page_table, pages_per_seq, 0);
    }
    const uint32_t dst = ring0 + (uint32_t)(iss_stage * stage_bytes);
    refill_pair_if(leader, bar0 + 8u * iss_stage, dst, ks, rbk, dst + kst, vs, rbv);
    ksrc += rbk;
    vsrc += rbv;
    ++iss_row;
    iss_stage = iss_stage + 1 == nstage ? 0 : iss_stage + 1;
  };
  int issued = min(n_loads, w.nstage);
  if (issued > 0 && rbk) {
    // the q~ fragments travel with the first stage: the previous item's reads of them are
    // ordered before the copy by the warp barrier and the proxy fence
    __syncwarp();
    fence_proxy_async_smem_if(leader);
    const uint32_t bar = smem_addr(&w.bars[0]);
    mbar_expect_tx_if(leader, bar, decode_qfrag_bytes<G>());  // stage 0's issue below arrives
    bulk_g2s_if(leader, smem_addr(w.qfrag), qt + kQtHeaderBytes, decode_qfrag_bytes<G>(), bar);
  }
  for (int k = 0; k < issued; ++k) issue_next();
  w.outstanding = issued;

  // wait for the next stage; returns its buffer or nullptr on timeout
  auto acquire = [&]() -> const uint8_t* {
    const uint32_t bar = bar0 + 8u * w.wait_stage, parity = (w.phase_bits >> w.wait_stage) & 1u;
    // the stage has normally landed already: one probe, and the bounded wait only when not
    if (!__all_sync(0xffffffffu, mbar_try_wait(bar, parity)) &&
        !__all_sync(0xffffffffu, mbar_wait_bounded(bar, parity, kWaitLimitNs)))
      return nullptr;
    w.phase_bits ^= 1u << w.wait_stage;
    return w.ring + (size_t)w.wait_stage * stage_bytes;
  };
  // release the stage just consumed and refill it with the next row pair of this item
  auto release = [&]() {
    __syncwarp();
    --w.outstanding;
    if (++w.wait_stage == w.nstage) w.wait_stage = 0;
    if (issued < n_loads) {
      issue_next();  // its proxy fence orders this warp's reads of the stage before the copies
      ++issued;
      ++w.outstanding;
    }
  };

  for (int row = row0; row < row1; ++row) {
    const uint8_t* buf = nullptr;
    if (n_loads) {
      buf = acquire();
      if (!buf) {
        w.failed = true;
        return;
      }
    }
    float s[8][NG][2];
    if (rbk) {
      if constexpr (BK > 0)
        k_row_scores<G, BK>(buf, kr, bfrag, qsum, qscale, one, s);
      else
        k_row_dispatch<G>(kb, buf, kr, bfrag, qsum, qscale, one, s);
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
    // row max per head; the reference max moves (and the accumulators are rescaled) only
    // when it is exceeded by more than kTau
    bool move = false;
    float alpha[NG];
#pragma unroll
    for (int u = 0; u < NG; ++u) {
      float mx = -INFINITY;
#pragma unroll
      for (int t = 0; t < 8; ++t) mx = fmaxf(mx, fmaxf(s[t][u][0], s[t][u][1]));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
      const bool mv = mx > mref[u] + kTau;
      alpha[u] = mv ? ex2_approx(mref[u] - mx) : 1.f;
      mref[u] = mv ? mx : mref[u];
      move |= mv;
    }
    if (__any_sync(0xffffffffu, move)) {
      for (int mu = 0; mu < ntile; ++mu) {
        float* o = osm + (mu * 32 + lane) * NO;
#pragma unroll
        for (int k = 0; k < NO; ++k) o[k] *= alpha[NG == 2 ? (k & 1) : 0];
      }
    }
    uint32_t bv[8][2];
    if constexpr (BV > 0) {
      row_probs<G, (BV <= 2 ? BV : 0)>(s, mref, bv);
      v_row_accumulate<G, BV>(buf + kst, vr, bv, one, osm);
    } else {
      if (vc == 1)
        row_probs<G, 1>(s, mref, bv);
      else if (vc == 2)
        row_probs<G, 2>(s, mref, bv);
      else
        row_probs<G, 0>(s, mref, bv);
      v_row_dispatch<G>(vbd, buf + kst, vr, bv, one, osm);
    }
    if (n_loads) release();
  }
  // ---- write the partial of this item: m, l and (O - c) 2^(10 - kmin) per query head ----
  __syncwarp();
  const int cr = vr & 15, ct = vr >> 4;  // constant rows r, r + 1: tile ct, rows cr, cr + 1
#pragma unroll
  for (int u = 0; u < NG; ++u) {
    const int g = Heads<G>::head(lane & 3, u);
    // entry of (row, head g) in a tile: lane 4 (row % 8) + column owner, slot by row half
    auto at = [&](int row) -> float {
      const int ln = 4 * (row & 7) + (G == 4 ? g : (g >> 1));
      const int sl = G == 4 ? ((row >> 3) & 1) : 2 * ((row >> 3) & 1) + (g & 1);
      return osm[(ct * 32 + ln) * NO + sl];
    };
    const float c = at(cr), l = at(cr + 1);
    float* pg = part + g * gstride;
    if ((lane >> 2) == 0) {
      pg[0] = mref[u];
      pg[1] = l;
    }
    for (int mu = 0; mu < ntile; ++mu) {
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

template <int G>
__global__ void __launch_bounds__(kDecodeWarps * 32, 4) decode_kernel(DecodeArgs a) {
  extern __shared__ __align__(128) uint8_t smem[];
  // the combine kernel may be scheduled as CTAs of this grid exit (it waits for the results)
  grid_dep_launch();
  const int warp = threadIdx.x >> 5;
  ScanWarp w;
  w.lane = threadIdx.x & 31;
  w.leader = w.lane == 0;
  w.ring_bytes = a.ring_bytes;
  const size_t warp_bytes = (size_t)w.ring_bytes + decode_osm_bytes<G>() + decode_qfrag_bytes<G>();
  w.ring = smem + (size_t)warp * warp_bytes;
  w.osm = reinterpret_cast<float*>(w.ring + w.ring_bytes);
  w.qfrag = reinterpret_cast<uint2*>(w.ring + w.ring_bytes + decode_osm_bytes<G>());
  w.bars = reinterpret_cast<uint64_t*>(smem + (size_t)kDecodeWarps * warp_bytes) + warp * kMaxStages;
  w.failed = false;
  w.phase_bits = 0;
  w.wait_stage = 0;
  w.nstage = 1;
  w.outstanding = 0;
  if (w.leader) {
    for (int i = 0; i < kMaxStages; ++i) mbar_init(smem_addr(&w.bars[i]), 1);
    fence_mbar_init();
  }
  __syncwarp();
  // the q~ blocks come from the query projection ahead, the cache from the appends before it
  grid_dep_wait();

  const WsHeader* wh = reinterpret_cast<const WsHeader*>(a.ws);
  const WsGroup* groups = reinterpret_cast<const WsGroup*>(a.ws + wh->groups_off);
  const WsItem* items = reinterpret_cast<const WsItem*>(a.ws + wh->items_off);
  const HeadEntry* heads = head_table(a.block);
  const int n_items = wh->n_items;
  // work items are taken in plan order from a shared counter, so that warps that finish early
  // take more (the items' costs differ with the heads' bit widths)
  unsigned int* next_item = const_cast<unsigned int*>(&wh->next_item);
  auto take = [&]() -> int {
    int v = 0;
    if (w.leader) v = (int)atomicAdd(next_item, 1u);
    return __shfl_sync(0xffffffffu, v, 0);
  };
  for (int item = take(); item < n_items && !w.failed; item = take()) {
    if constexpr (G == 4) {
      // the bit widths of 1 to 3 that carry most of the cache at low rates, and the 3- to 5-bit
      // pairs of rates of 3 to 4 bpd, get their own code
      const WsGroup gr = groups[items[item].group];
      const HeadEntry hk = heads[gr.k_head], hv = heads[gr.v_head];
      const int key = (hk.r > 0 ? hk.b : 0) * 16 + (hv.r > 0 ? hv.b : 0);
      switch (key) {
        case 0x11: scan_item<G, 1, 1>(a, w, item); break;
        case 0x12: scan_item<G, 1, 2>(a, w, item); break;
        case 0x13: scan_item<G, 1, 3>(a, w, item); break;
        case 0x21: scan_item<G, 2, 1>(a, w, item); break;
        case 0x22: scan_item<G, 2, 2>(a, w, item); break;
        case 0x23: scan_item<G, 2, 3>(a, w, item); break;
        case 0x31: scan_item<G, 3, 1>(a, w, item); break;
        case 0x32: scan_item<G, 3, 2>(a, w, item); break;
        case 0x33: scan_item<G, 3, 3>(a, w, item); break;
        case 0x34: scan_item<G, 3, 4>(a, w, item); break;
        case 0x43: scan_item<G, 4, 3>(a, w, item); break;
        case 0x44: scan_item<G, 4, 4>(a, w, item); break;
        case 0x45: scan_item<G, 4, 5>(a, w, item); break;
        case 0x54: scan_item<G, 5, 4>(a, w, item); break;
        case 0x55: scan_item<G, 5, 5>(a, w, item); break;
        default: scan_item<G, 0, 0>(a, w, item); break;
      }
    } else {
      // G = 8 (low rates: the 1- and 2-bit pairs carry nearly all of the cache)
      const WsGroup gr = groups[items[item].group];
      const HeadEntry hk = heads[gr.k_head], hv = heads[gr.v_head];
      const int key = (hk.r > 0 ? hk.b : 0) * 16 + (hv.r > 0 ? hv.b : 0);
      switch (key) {
        case 0x11: scan_item<G, 1, 1>(a, w, item); break;
        case 0x12: scan_item<G, 1, 2>(a, w, item); break;
        case 0x21: scan_item<G, 2, 1>(a, w, item); break;
        case 0x22: scan_item<G, 2, 2>(a, w, item); break;
        default: scan_item<G, 0, 0>(a, w, item); break;
      }
    }
  }
  if (w.failed) {
    if (w.leader) atomicOr(&g_status, 1u);
    // drain the copies still in flight before the shared memory goes away
    for (int k = 0; k < w.outstanding; ++k) {
      if (!mbar_wait_bounded(smem_addr(&w.bars[w.wait_stage]), (w.phase_bits >> w.wait_stage) & 1u, kWaitLimitNs))
        break;
      w.phase_bits ^= 1u << w.wait_stage;
      if (++w.wait_stage == w.nstage) w.wait_stage = 0;
    }
  }
  // the last CTA to run out of items puts the work counter back to 0 for the next launch:
  // by then every warp of the grid has taken its final (empty) index
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned int* done = const_cast<unsigned int*>(&wh->done_ctas);
    if (atomicAdd(done, 1u) == gridDim.x - 1) {
      atomicExch(next_item, 0u);
      atomicExch(done, 0u);
    }
  }
}

}  // namespace cobra
