// Decode attention for models with the rotary position embedding (RoPE).
//
// The paper compresses K before the rotation (Sec. 5, "Scope"; App. "Post-RoPE experiments":
// after it the per-head covariance depends on the position), so such a model attends with
// every reconstructed key turned to its own position t and the query to its position p:
//   s_t = <R(p) q, R(t) K^_t> / sqrt(d),   K^_t = mu_K + W_K Delta_K (c_t - 2^{b-1} + 1/2),
// R(x) turning channel pair (j, j + d/2) by the angle x omega_j, omega_j = theta^(-2j/d).
// R(t) differs per token, so W_K cannot be folded into one projected query as in the rank-
// space scan of decode.cuh: each key is rebuilt in the d-dimensional space on the tensor
// cores, turned, and scored.
//
// Channel order.  Inside these kernels, channel position P = 2j + e holds model channel
// j + e d/2 (the pairs interleaved), so that the two halves of a pair sit side by side in an
// MMA accumulator lane and the rotation stays in registers.  W_K's rows and the query are
// permuted alike; the dot product does not depend on the order.
//
//   rope_table_kernel  cos and sin of x omega_j in fp64, for x = i < 16 (fine rows) and
//                      x = 16 m (coarse rows); any position x = 16 m + i composes from one of
//                      each by the angle-addition formulas.
//   rope_qprep_kernel  q' = (Delta_K / sqrt d) log2(e) R(p) q per query head, scaled by a
//                      power of two, split into fp16 hi + lo and laid out as the score MMA's
//                      B fragments in the workspace's q~ block of the group.
//   rope_scan_kernel   CTAs take whole (seq, layer, kv head) groups of the decode plan; the
//                      CTA's warps share the group's rows.  Per pair of 16-token tiles:
//                        rebuild  X = seed + A W'   (A the unpacked codes, W' = W_K^T hi + lo)
//                        turn     X <- R(t) X       (the token's composed angle, per pair)
//                        score    S += X q'         (X and q' both split hi + lo)
//                      followed by the scan's online softmax and rank-space accumulation of
//                      V (not rotated), and a merge of the CTA's warps into the first of the
//                      group's partial slots (the others are left empty for combine_kernel).
//   combine_kernel     (decode_heads.cuh) as for the plain decode.
//
// The codes unpack to A = 1 + c 2^(k - 10) with the per-register window k of the scan (see
// Window).  With seed_k = 2^(k-10) (mu'/Delta - (2^{b-1} - 1/2) W'1) - W'1 the product gives
// X = 2^(k-10) K^'/Delta exactly (K^' = K^ in the interleaved order), and the score's factor
// Delta 2^(10-k) / sqrt(d) is applied after the MMA.  A head with r_K = 0 has X = mu' (Delta
// taken as 1 on both sides).
#pragma once

#include "decode.cuh"

namespace cobra {

constexpr int kRopeFine = 16;         // positions per coarse step (fine rows 0..15)
constexpr int kRopeRowFloats = 128;   // floats per table row: [jj 4][n 16][cos, sin]
constexpr int kRopeMaxWarps = 8;
constexpr int kRopeKTiles = 8;        // channel tiles of 16 (r <= 128)
constexpr int kRopeSeedSlots = 8;     // windows k = 2 .. 9
constexpr int kRopeMergeStride = 4 + kD;  // floats per query head in a warp's partial
constexpr int kRopeCh = 4;            // blocks of 16 positions rebuilt per pass over the codes

// Table entry of pair j = 4 n + jj within a row: [(jj * 16 + n) * 2 + (0: cos, 1: sin)].  The
// two pairs (8 ch + jj, 8 ch + 4 + jj) that a lane turns in channel block ch are one float4.
__host__ __device__ constexpr int rope_entry(int j) { return ((j & 3) * 16 + (j >> 2)) * 2; }

__host__ __device__ constexpr size_t rope_table_floats(int n_coarse) {
  return (size_t)(kRopeFine + n_coarse) * kRopeRowFloats;
}

struct RopeArgs {
  const float* table;  // [kRopeFine + n_coarse][kRopeRowFloats]
  const int* q_pos;    // [n_seqs] query positions, or null: seq_len - 1
  int n_coarse;        // positions < 16 n_coarse are covered
  int stage_bytes;     // per-warp staging stage: channel tiles of a K row + a V row
};

constexpr size_t kRopeWfragBytes = (size_t)kRopeKTiles * 16 * 2 * 32 * 8;
constexpr size_t kRopeSeedBytes = (size_t)kRopeSeedSlots * kD * sizeof(float);
constexpr size_t kRopeFineBytes = (size_t)kRopeFine * kRopeRowFloats * sizeof(float);
template <int G>
__host__ __device__ constexpr size_t rope_fixed_bytes() {
  return kRopeWfragBytes + kRopeSeedBytes + kRopeFineBytes + decode_qfrag_bytes<G>();
}
template <int G>
__host__ __device__ constexpr size_t rope_warp_bytes(int stage_bytes) {
  return 2 * (size_t)stage_bytes + decode_osm_bytes<G>();
}

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_1() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_0() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

// (cos, sin) of x omega_j for x = 16 m + i from the coarse (m) and fine (i) entries
__device__ __forceinline__ void rope_compose(float cm, float sm, float ci, float si, float& c, float& s) {
  c = fmaf(cm, ci, -sm * si);
  s = fmaf(sm, ci, cm * si);
}

// fp16 hi + lo parts of two values, packed as the MMA's f16x2 operands
__device__ __forceinline__ void split_f16x2(float a, float b, uint32_t& hi, uint32_t& lo) {
  const __half2 h = __floats2half2_rn(a, b);
  const float2 f = __half22float2(h);
  const __half2 l = __floats2half2_rn(a - f.x, b - f.y);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = *reinterpret_cast<const uint32_t*>(&l);
}

// ---------------------------------------------------------------------------------------
// Angle tables: row x < 16 holds position x, row 16 + m position 16 m (fp64 angles, rounded
// once to fp32).
// ---------------------------------------------------------------------------------------
__global__ void rope_table_kernel(float* table, int n_rows, double theta) {
  // an earlier decode may still read the table being overwritten
  grid_dep_wait();
  grid_dep_launch();
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= n_rows * (kD / 2)) return;
  const int x = idx / (kD / 2), j = idx % (kD / 2);
  const double pos = x < kRopeFine ? (double)x : 16.0 * (double)(x - kRopeFine);
  const double om = pow(theta, -2.0 * (double)j / (double)kD);
  double s, c;
  sincos(pos * om, &s, &c);
  float* e = table + (size_t)x * kRopeRowFloats + rope_entry(j);
  e[0] = (float)c;
  e[1] = (float)s;
}

// ---------------------------------------------------------------------------------------
// Query preparation: one CTA per (layer, kv head), one warp per sequence at a time.
// ---------------------------------------------------------------------------------------
template <int G>
__global__ void __launch_bounds__(kHeadThreads) rope_qprep_kernel(DecodeArgs a, RopeArgs ra) {
  grid_dep_launch();
  constexpr int NTK = Heads<G>::NTK, NW = kHeadThreads / 32;
  __shared__ __align__(16) float qr[NW][G * kD];  // turned, scaled query of the warp's sequence
  const WsHeader* wh = reinterpret_cast<const WsHeader*>(a.ws);
  const WsGroup* groups = reinterpret_cast<const WsGroup*>(a.ws + wh->groups_off);
  grid_dep_wait();
  const int S = wh->n_seqs;
  const int* hg = reinterpret_cast<const int*>(a.ws + wh->hg_off) + (size_t)blockIdx.x * S;
  const WsGroup g0 = groups[hg[0]];
  const HeadEntry hk = head_table(a.block)[g0.k_head];
  const int layer = g0.layer, kv = g0.kv;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float dk = (hk.r > 0 && hk.delta > 0.f) ? hk.delta : 1.f;
  const float fac = dk * 0.088388347648318440f * 1.4426950408889634f;  // Delta/sqrt(128)*log2(e)
  const int max_pos = kRopeFine * ra.n_coarse;
  float* Q = qr[warp];
  for (int s = warp; s < S; s += NW) {
    const int T = a.seq_lens[s];
    int p = ra.q_pos ? ra.q_pos[s] : T - 1;
    // an empty sequence (default position -1) has no output; any other position outside
    // the table is reported and clamped
    const bool bad = p < 0 ? (ra.q_pos != nullptr) : p >= max_pos;
    if (bad && lane == 0) atomicOr(&g_status, 2u);
    p = min(max(p, 0), max_pos - 1);
    const float* fine = ra.table + (size_t)(p & 15) * kRopeRowFloats;
    const float* coarse = ra.table + (size_t)(kRopeFine + (p >> 4)) * kRopeRowFloats;
    float cj[2], sj[2];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int e = rope_entry(lane + 32 * h);
      rope_compose(coarse[e], coarse[e + 1], fine[e], fine[e + 1], cj[h], sj[h]);
    }
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const __nv_bfloat16* qp = a.q + layer * a.q_sl + (long long)s * a.q_ss + (long long)(kv * G + g) * kD;
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int j = lane + 32 * h;
        const float xa = __bfloat162float(qp[j]), xb = __bfloat162float(qp[j + kD / 2]);
        Q[g * kD + 2 * j] = fac * fmaf(xa, cj[h], -xb * sj[h]);
        Q[g * kD + 2 * j + 1] = fac * fmaf(xa, sj[h], xb * cj[h]);
      }
    }
    __syncwarp();
    float amax = 0.f;
    for (int i = lane; i < G * kD; i += 32) amax = fmaxf(amax, fabsf(Q[i]));
#pragma unroll
    for (int m = 16; m; m >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, m));
    int e = 0;
    if (amax > 0.f) {
      int ex;
      frexpf(amax, &ex);  // amax = m 2^ex, m in [0.5, 1): scaled into [256, 512)
      e = 9 - ex;
    }
    const float up = ldexpf(1.f, e);
    unsigned char* qt = a.ws + wh->qt_off + (size_t)hg[s] * wh->qt_stride;
    float* qhdr = reinterpret_cast<float*>(qt);
    if (lane < 8) qhdr[lane] = 0.f;
    if (lane == 8) qhdr[8] = ldexpf(1.f, -e);
    // element (k, n) of fragment (kappa, nt) = hi or lo part of q' at position 16 kappa + k
    // for the query head of column n (see Heads)
    uint2* frag = reinterpret_cast<uint2*>(qt + kQtHeaderBytes);
    for (int idx = lane; idx < 8 * NTK * 32; idx += 32) {
      const int fl = idx & 31, nt = (idx >> 5) % NTK, kap = idx / (32 * NTK);
      const int j = fl & 3, n = fl >> 2;
      const int g = Heads<G>::col_head(nt, n), lo = Heads<G>::col_lo(nt, n);
      const int ks[4] = {2 * j, 2 * j + 1, 2 * j + 8, 2 * j + 9};
      float e4[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float x = Q[g * kD + 16 * kap + ks[u]] * up;
        const float h = __half2float(__float2half_rn(x));
        e4[u] = lo ? (x - h) : h;
      }
      frag[(kap * NTK + nt) * 32 + fl] = make_uint2(pack_f16(e4[0], e4[1]), pack_f16(e4[2], e4[3]));
    }
    __syncwarp();
  }
}

// ---------------------------------------------------------------------------------------
// K side: scores of one 128-token code row (log2 units) for the lane's query heads, laid out
// as k_row_scores lays them out: s[t][u][0] for token 16 t + lane/4, s[t][u][1] for + 8.
// B = 0 stands for a head without K codes (r_K = 0).
//   wfrag  W' B fragments [kt][n-tile][hi, lo][lane] (channels past r are zero)
//   seed4  [slot][ch][jj] float4: positions 16 ch + 2 jj + {0, 1, 8, 9} of window slot k - 2
//   fine4  fine table entries as float4 [jj][ch][i]; coarse4 the coarse rows (global)
//   crow   coarse row of the row's first token tile (token 128 row -> 8 row)
// ---------------------------------------------------------------------------------------
template <int B>
__host__ __device__ constexpr int rope_slot(int rho) {
  return B > 0 ? Window<B>::k(rho) - 2 : 0;
}
template <int B>
__host__ __device__ constexpr float rope_unscale(int rho) {
  return B > 0 ? Window<B>::inv_scale(rho) : 1.f;
}

template <int G, int B>
__device__ __forceinline__ void rope_k_row(const uint8_t* stage, int rk, int crow, int n_coarse,
                                           const float4* __restrict__ coarse4, const uint2* wfrag,
                                           const float4* seed4, const float4* fine4, const uint2* qfrag,
                                           float qscale, uint32_t one, float (&s)[8][G / 4][2]) {
  constexpr int NTK = Heads<G>::NTK, NG = Heads<G>::NG;
  constexpr int BB = B > 0 ? B : 1;
  const int lane = threadIdx.x & 31, jj = lane & 3, gi = lane >> 2;
  const int nk = B > 0 ? (rk + 15) >> 4 : 0;
  // lane's pieces: strips 8 kt + jj and + 4, piece gi (the scan's K-row A fragments)
  const uint8_t* pa = stage + jj * 32 * BB + gi * 4 * BB;
#pragma unroll
  for (int mp = 0; mp < 4; ++mp) {
    float sacc[2][NTK][4];
#pragma unroll
    for (int mi = 0; mi < 2; ++mi)
#pragma unroll
      for (int nt = 0; nt < NTK; ++nt) sacc[mi][nt][0] = sacc[mi][nt][1] = sacc[mi][nt][2] = sacc[mi][nt][3] = 0.f;
    const float4* co[2];
#pragma unroll
    for (int mi = 0; mi < 2; ++mi) co[mi] = coarse4 + (size_t)min(crow + 2 * mp + mi, n_coarse - 1) * (kRopeRowFloats / 4);
#pragma unroll 1
    for (int ch0 = 0; ch0 < 8; ch0 += kRopeCh) {
      // rebuild X for n-tiles 2 ch, 2 ch + 1 (ch = ch0 .. ch0 + kRopeCh - 1) of both token
      // tiles, starting from the seeds
      float x[2][kRopeCh][2][4];
#pragma unroll
      for (int mi = 0; mi < 2; ++mi) {
        const int t = 2 * mp + mi;
#pragma unroll
        for (int c = 0; c < kRopeCh; ++c) {
          const float4 sl = seed4[(rope_slot<B>(2 * t) * 8 + ch0 + c) * 4 + jj];
          const float4 sh = seed4[(rope_slot<B>(2 * t + 1) * 8 + ch0 + c) * 4 + jj];
          x[mi][c][0][0] = sl.x;
          x[mi][c][0][1] = sl.y;
          x[mi][c][0][2] = sh.x;
          x[mi][c][0][3] = sh.y;
          x[mi][c][1][0] = sl.z;
          x[mi][c][1][1] = sl.w;
          x[mi][c][1][2] = sh.z;
          x[mi][c][1][3] = sh.w;
        }
      }
      if constexpr (B > 0) {
        // the codes of both token tiles are unpacked again for every kRopeCh blocks of 16
        // positions: holding them for all channel tiles would not fit the registers
#pragma unroll 2
        for (int kt = 0; kt < nk; ++kt) {
          uint32_t wa[B], wb[B];
          load_piece<B>(pa + kt * 8 * 32 * B, wa);
          load_piece<B>(pa + kt * 8 * 32 * B + 4 * 32 * B, wb);
          uint32_t av[2][4];
#pragma unroll
          for (int mi = 0; mi < 2; ++mi) {
            const int t = 2 * mp + mi;
            av[mi][0] = unpack_reg<B>(wa, 2 * t, one);
            av[mi][1] = unpack_reg<B>(wa, 2 * t + 1, one);
            av[mi][2] = unpack_reg<B>(wb, 2 * t, one);
            av[mi][3] = unpack_reg<B>(wb, 2 * t + 1, one);
          }
#pragma unroll
          for (int c = 0; c < kRopeCh; ++c) {
            const uint2* wf = wfrag + (size_t)((kt * 16 + 2 * (ch0 + c)) * 2) * 32 + lane;
            const uint2 bw[2][2] = {{wf[0], wf[32]}, {wf[64], wf[96]}};  // [n-tile][hi, lo]
            // the hi and lo products of an accumulator are issued four MMAs apart
#pragma unroll
            for (int limb = 0; limb < 2; ++limb)
#pragma unroll
              for (int mi = 0; mi < 2; ++mi)
#pragma unroll
                for (int nn = 0; nn < 2; ++nn)
                  mma_f16(x[mi][c][nn], av[mi][0], av[mi][1], av[mi][2], av[mi][3], bw[nn][limb].x, bw[nn][limb].y);
          }
        }
      }
#pragma unroll
      for (int c = 0; c < kRopeCh; ++c) {
        const int ch = ch0 + c;
        // turn each pair (x[..][2h], x[..][2h+1]) by its token's angle: pair 8 ch + jj in
        // n-tile 2 ch, 8 ch + 4 + jj in n-tile 2 ch + 1; token row gi (h = 0) or gi + 8 (h = 1)
        const float4 f0 = fine4[(jj * 8 + ch) * kRopeFine + gi], f1 = fine4[(jj * 8 + ch) * kRopeFine + gi + 8];
#pragma unroll
        for (int mi = 0; mi < 2; ++mi) {
          const float4 cm = __ldg(co[mi] + jj * 8 + ch);
#pragma unroll
          for (int nn = 0; nn < 2; ++nn) {
            const float c0 = nn ? cm.z : cm.x, s0 = nn ? cm.w : cm.y;
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const float4 f = h ? f1 : f0;
              float cs, sn;
              rope_compose(c0, s0, nn ? f.z : f.x, nn ? f.w : f.y, cs, sn);
              const float xa = x[mi][c][nn][2 * h], xb = x[mi][c][nn][2 * h + 1];
              x[mi][c][nn][2 * h] = fmaf(xa, cs, -xb * sn);
              x[mi][c][nn][2 * h + 1] = fmaf(xa, sn, xb * cs);
            }
          }
        }
        // the two n-tiles' accumulators are the A fragment of the k-tile of positions
        // 16 ch .. 16 ch + 15 for the score MMA against q' (hi and lo of both sides)
        uint2 bq[NTK];
#pragma unroll
        for (int nt = 0; nt < NTK; ++nt) bq[nt] = qfrag[(ch * NTK + nt) * 32 + lane];
#pragma unroll
        for (int mi = 0; mi < 2; ++mi) {
          uint32_t h[4], l[4];
          split_f16x2(x[mi][c][0][0], x[mi][c][0][1], h[0], l[0]);
          split_f16x2(x[mi][c][0][2], x[mi][c][0][3], h[1], l[1]);
          split_f16x2(x[mi][c][1][0], x[mi][c][1][1], h[2], l[2]);
          split_f16x2(x[mi][c][1][2], x[mi][c][1][3], h[3], l[3]);
#pragma unroll
          for (int nt = 0; nt < NTK; ++nt) {
            mma_f16(sacc[mi][nt], h[0], h[1], h[2], h[3], bq[nt].x, bq[nt].y);
            mma_f16(sacc[mi][nt], l[0], l[1], l[2], l[3], bq[nt].x, bq[nt].y);
          }
        }
      }
    }
    // hi + lo columns of each head, times Delta 2^(10 - k) / sqrt(d) log2(e) 2^-e
#pragma unroll
    for (int mi = 0; mi < 2; ++mi) {
      const int t = 2 * mp + mi;
      const float sc0 = qscale * rope_unscale<B>(2 * t), sc1 = qscale * rope_unscale<B>(2 * t + 1);
#pragma unroll
      for (int u = 0; u < NG; ++u) {
        const float v0 = G == 4 ? sacc[mi][0][0] + sacc[mi][0][1] : sacc[mi][0][u] + sacc[mi][NTK - 1][u];
        const float v1 = G == 4 ? sacc[mi][0][2] + sacc[mi][0][3] : sacc[mi][0][2 + u] + sacc[mi][NTK - 1][2 + u];
        s[t][u][0] = v0 * sc0;
        s[t][u][1] = v1 * sc1;
      }
    }
  }
}

template <int G>
__device__ __forceinline__ void rope_k_dispatch(int b, const uint8_t* stage, int rk, int crow, int n_coarse,
                                                const float4* coarse4, const uint2* wfrag, const float4* seed4,
                                                const float4* fine4, const uint2* qfrag, float qscale, uint32_t one,
                                                float (&s)[8][G / 4][2]) {
  if (rk == 0) {
    rope_k_row<G, 0>(stage, rk, crow, n_coarse, coarse4, wfrag, seed4, fine4, qfrag, qscale, one, s);
    return;
  }
  switch (b) {
    case 1: rope_k_row<G, 1>(stage, rk, crow, n_coarse, coarse4, wfrag, seed4, fine4, qfrag, qscale, one, s); break;
    case 2: rope_k_row<G, 2>(stage, rk, crow, n_coarse, coarse4, wfrag, seed4, fine4, qfrag, qscale, one, s); break;
    case 3: rope_k_row<G, 3>(stage, rk, crow, n_coarse, coarse4, wfrag, seed4, fine4, qfrag, qscale, one, s); break;
    case 4: rope_k_row<G, 4>(stage, rk, crow, n_coarse, coarse4, wfrag, seed4, fine4, qfrag, qscale, one, s); break;
    case 5: rope_k_row<G, 5>(stage, rk, crow, n_coarse, coarse4, wfrag, seed4, fine4, qfrag, qscale, one, s); break;
    case 6: rope_k_row<G, 6>(stage, rk, crow, n_coarse, coarse4, wfrag, seed4, fine4, qfrag, qscale, one, s); break;
    case 7: rope_k_row<G, 7>(stage, rk, crow, n_coarse, coarse4, wfrag, seed4, fine4, qfrag, qscale, one, s); break;
    default: rope_k_row<G, 8>(stage, rk, crow, n_coarse, coarse4, wfrag, seed4, fine4, qfrag, qscale, one, s); break;
  }
}

// Copy n bytes (a multiple of 16) from global to shared memory, 16 bytes per lane and step.
__device__ __forceinline__ void warp_copy_async(uint8_t* dst, const uint8_t* src, uint32_t n, int lane) {
  for (uint32_t o = 16u * lane; o < n; o += 512u) cp_async16(smem_addr(dst + o), src + o);
}

// ---------------------------------------------------------------------------------------
// The scan: one CTA per SM takes (seq, layer, kv head) groups from the plan's counter (W_K is
// staged once per group, and whole groups keep the warps' shares of rows even); its warps take
// the group's rows in turn, each with its own softmax state and V accumulators, and the warps'
// partials are merged into the group's first slot.
// ---------------------------------------------------------------------------------------
template <int G>
__global__ void __launch_bounds__(kRopeMaxWarps * 32, 1) rope_scan_kernel(DecodeArgs a, RopeArgs ra) {
  constexpr int NG = G / 4, NO = OAcc<G>::N;
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ int s_item;
  // the combine kernel may be scheduled as CTAs of this grid exit (it waits for the results)
  grid_dep_launch();
  uint2* wfrag = reinterpret_cast<uint2*>(smem);
  float4* seed4 = reinterpret_cast<float4*>(smem + kRopeWfragBytes);
  float4* fine4 = reinterpret_cast<float4*>(smem + kRopeWfragBytes + kRopeSeedBytes);
  uint2* qfrag = reinterpret_cast<uint2*>(smem + kRopeWfragBytes + kRopeSeedBytes + kRopeFineBytes);
  const int nw = blockDim.x >> 5, warp = threadIdx.x >> 5, lane = threadIdx.x & 31, tid = threadIdx.x;
  uint8_t* wst = smem + rope_fixed_bytes<G>() + (size_t)warp * rope_warp_bytes<G>(ra.stage_bytes);
  float* osm = reinterpret_cast<float*>(wst + 2 * (size_t)ra.stage_bytes);
  // the q' blocks come from the query preparation ahead, the cache from the appends before it
  grid_dep_wait();

  const WsHeader* wh = reinterpret_cast<const WsHeader*>(a.ws);
  const WsGroup* groups = reinterpret_cast<const WsGroup*>(a.ws + wh->groups_off);
  const HeadEntry* heads = head_table(a.block);
  const float* pool = param_pool(a.block);
  float* parts = reinterpret_cast<float*>(a.ws + wh->part_off);
  const int n_groups = wh->n_groups, gstride = wh->g_stride, pstride = wh->part_stride;
  unsigned int* next_item = const_cast<unsigned int*>(&wh->next_item);
  const float4* coarse4 = reinterpret_cast<const float4*>(ra.table + (size_t)kRopeFine * kRopeRowFloats);
  // fine rows in shared memory as [jj][ch][i] float4, so that the lanes of a warp (token i =
  // lane / 4 or + 8, pair group jj = lane % 4) read distinct banks
  for (int idx = tid; idx < (int)(kRopeFineBytes / 16); idx += blockDim.x) {
    const int i = idx / 32, q = idx % 32;  // table float4 q = jj * 8 + ch of fine row i
    fine4[q * kRopeFine + i] = reinterpret_cast<const float4*>(ra.table)[idx];
  }
  const uint32_t one = a.one;
  int staged_head = -1;

  for (;;) {
    if (tid == 0) s_item = (int)atomicAdd(next_item, 1u);
    __syncthreads();  // (also: every warp is done with the previous group's shared memory)
    const int grp = s_item;
    if (grp >= n_groups) break;
    const WsGroup gr = groups[grp];
    const HeadEntry hk = heads[gr.k_head], hv = heads[gr.v_head];
    const int rk = hk.r, kb = hk.b, vr = hv.r, vb = hv.b;
    const int nk = (rk + 15) >> 4;
    if (gr.k_head != staged_head) {
      staged_head = gr.k_head;
      const float* W = pool + hk.w_off;  // d x r, column c at W + c d
      // W' fragments: element (k, n) of (kt, n-tile) = W_K[model channel of position 8 nt + n][16 kt + k]
      for (int idx = tid; idx < nk * 16 * 2 * 32; idx += blockDim.x) {
        const int ln = idx & 31, limb = (idx >> 5) & 1, nt = (idx >> 6) & 15, kt = idx >> 10;
        const int P = 8 * nt + (ln >> 2), dm = (P >> 1) + (P & 1) * (kD / 2);
        const int c0 = 16 * kt + 2 * (ln & 3);
        const int cs[4] = {c0, c0 + 1, c0 + 8, c0 + 9};
        float v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const float w = cs[u] < rk ? W[(size_t)cs[u] * kD + dm] : 0.f;
          const float h = __half2float(__float2half_rn(w));
          v[u] = limb ? (w - h) : h;
        }
        wfrag[idx] = make_uint2(pack_f16(v[0], v[1]), pack_f16(v[2], v[3]));
      }
      // seeds of every window slot: 2^(k-10) (mu'/Delta - c_b W'1) - W'1, or mu' when r = 0
      // (one warp per position: the lanes sum W'1 over the channels, lane k - 2 writes slot k)
      float* seed = reinterpret_cast<float*>(seed4);
      for (int P = warp; P < kD; P += nw) {
        const int dm = (P >> 1) + (P & 1) * (kD / 2);
        float w1 = 0.f;
        for (int c = lane; c < rk; c += 32) w1 += W[(size_t)c * kD + dm];
#pragma unroll
        for (int o = 16; o; o >>= 1) w1 += __shfl_xor_sync(0xffffffffu, w1, o);
        if (lane < kRopeSeedSlots) {
          const float mu = pool[hk.mu_off + dm];
          const float base = rk > 0 ? mu / hk.delta - ((float)(1 << (kb - 1)) - 0.5f) * w1 : 0.f;
          const int ch = P >> 4, hi8 = (P >> 3) & 1, jq = (P >> 1) & 3, e = P & 1;
          const float v = rk > 0 ? ldexpf(base, lane + 2 - 10) - w1 : (lane == 0 ? mu : 0.f);
          seed[((lane * 8 + ch) * 4 + jq) * 4 + 2 * hi8 + e] = v;
        }
      }
    }
    const unsigned char* qt = a.ws + wh->qt_off + (size_t)grp * wh->qt_stride;
    for (int i = tid; i < (int)(decode_qfrag_bytes<G>() / 16); i += blockDim.x)
      reinterpret_cast<uint4*>(qfrag)[i] = reinterpret_cast<const uint4*>(qt + kQtHeaderBytes)[i];
    const float qscale = reinterpret_cast<const float*>(qt)[8];
    __syncthreads();

    // ---- this warp's rows of the group: rows warp, warp + nw, ... (never past the cache's
    //      rows of a sequence) ----
    const int T = a.seq_lens[gr.seq];
    const int rows_valid = (T + kRowTokens - 1) / kRowTokens;
    const int row0 = 0, row1 = min(rows_valid, a.page_table ? 2 * a.pages_per_seq : a.rows_per_seq);
    const uint32_t rbk = rk > 0 ? 16u * rk * kb : 0u, rbv = vr > 0 ? 16u * vr * vb : 0u;
    const uint32_t kst = rk > 0 ? 256u * kb * nk : 0u;  // whole channel tiles (the last may read past the row)
    const bool fits = kst + ((rbv + 127u) & ~127u) <= (uint32_t)ra.stage_bytes;
    if (!fits && tid == 0) atomicOr(&g_status, 2u);
    if (T > kRopeFine * ra.n_coarse && tid == 0) atomicOr(&g_status, 2u);  // positions past the table
    const int ntile = (vr >> 4) + 1;
    for (int k = 0; k < ntile * NO; ++k) osm[k * 32 + lane] = 0.f;
    float mref[NG];
#pragma unroll
    for (int u = 0; u < NG; ++u) mref[u] = -INFINITY;
    const int vc = (vr > 0 && vb <= 2) ? vb : 0;
    const int vbd = vr > 0 ? vb : 0;
    const float vout = vr == 0 ? 0.f : (float)(1 << (vb == 1 ? 5 : vb == 2 ? 6 : vb));
    const uint8_t* kbase = a.cache + hk.cache_off;
    const uint8_t* vbase = a.cache + hv.cache_off;
    auto issue = [&](int row, int st) {
      if (fits && row < row1) {
        uint8_t* dst = wst + (size_t)st * ra.stage_bytes;
        if (rbk)
          warp_copy_async(dst, kbase + row_offset(0, rbk, gr.seq, row, a.page_table, a.pages_per_seq, a.rows_per_seq),
                          rbk, lane);
        if (rbv)
          warp_copy_async(dst + kst,
                          vbase + row_offset(0, rbv, gr.seq, row, a.page_table, a.pages_per_seq, a.rows_per_seq),
                          rbv, lane);
      }
      cp_async_commit();
    };
    issue(row0 + warp, 0);
    issue(row0 + warp + nw, 1);
    int k = 0;
    for (int row = row0 + warp; fits && row < row1; row += nw, ++k) {
      cp_async_wait_1();
      __syncwarp();
      const uint8_t* buf = wst + (size_t)(k & 1) * ra.stage_bytes;
      float s[8][NG][2];
      rope_k_dispatch<G>(kb, buf, rk, 8 * row, ra.n_coarse, coarse4, wfrag, seed4, fine4, qfrag, qscale, one, s);
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
          for (int q = 0; q < NO; ++q) o[q] *= alpha[NG == 2 ? (q & 1) : 0];
        }
      }
      uint32_t bv[8][2];
      if (vc == 1)
        row_probs<G, 1>(s, mref, bv);
      else if (vc == 2)
        row_probs<G, 2>(s, mref, bv);
      else
        row_probs<G, 0>(s, mref, bv);
      v_row_dispatch<G>(vbd, buf + kst, vr, bv, one, osm);
      __syncwarp();  // every lane is done with the stage before it is refilled
      issue(row + 2 * nw, k & 1);
    }
    cp_async_wait_0();
    __syncwarp();
    // ---- the warp's partial (m, l, (O - c) 2^(10 - kmin)) into its staging area ----
    float* mg = reinterpret_cast<float*>(wst);
    const int cr = vr & 15, ct = vr >> 4;
#pragma unroll
    for (int u = 0; u < NG; ++u) {
      const int g = Heads<G>::head(lane & 3, u);
      auto at = [&](int r) -> float {
        const int ln = 4 * (r & 7) + (G == 4 ? g : (g >> 1));
        const int sl = G == 4 ? ((r >> 3) & 1) : 2 * ((r >> 3) & 1) + (g & 1);
        return osm[(ct * 32 + ln) * NO + sl];
      };
      const float c = at(cr), l = at(cr + 1);
      float* pg = mg + g * kRopeMergeStride;
      if ((lane >> 2) == 0) {
        pg[0] = mref[u];
        pg[1] = l;
      }
      for (int mu = 0; mu < ntile; ++mu) {
        const float* o = osm + (mu * 32 + lane) * NO;
        const float o0 = NO == 2 ? o[0] : o[u], o1 = NO == 2 ? o[1] : o[2 + u];
        const int ch0 = 16 * mu + (lane >> 2), ch1 = ch0 + 8;
        if (ch0 < vr) pg[4 + ch0] = (o0 - c) * vout;
        if (ch1 < vr) pg[4 + ch1] = (o1 - c) * vout;
      }
    }
    __syncthreads();
    // ---- merge the warps into the group's first slot: m = max m_w, l = sum 2^(m_w - m) l_w,
    //      O likewise; the group's other slots are left empty (m = -inf, l = 0, O = 0) ----
    for (int idx = tid; idx < (gr.n_items - 1) * G * (1 + vr); idx += blockDim.x) {
      const int k = 1 + idx / (G * (1 + vr)), rem = idx % (G * (1 + vr)), g = rem / (1 + vr), e = rem % (1 + vr);
      float* pg = parts + (size_t)(gr.first_item + k) * pstride + g * gstride;
      if (e == 0) {
        pg[0] = -INFINITY;
        pg[1] = 0.f;
      } else {
        pg[3 + e] = 0.f;
      }
    }
    float* part = parts + (size_t)gr.first_item * pstride;
    const size_t wb = rope_warp_bytes<G>(ra.stage_bytes) / sizeof(float);
    const float* mg0 = reinterpret_cast<const float*>(smem + rope_fixed_bytes<G>());
    for (int idx = tid; idx < G * (1 + vr); idx += blockDim.x) {
      const int g = idx / (1 + vr), e = idx % (1 + vr);
      float m = -INFINITY;
      for (int w = 0; w < nw; ++w) m = fmaxf(m, mg0[w * wb + g * kRopeMergeStride]);
      float acc = 0.f;
      if (m != -INFINITY) {
        for (int w = 0; w < nw; ++w) {
          const float* pw = mg0 + w * wb + g * kRopeMergeStride;
          if (pw[0] != -INFINITY) acc += exp2f(pw[0] - m) * (e == 0 ? pw[1] : pw[3 + e]);
        }
      }
      float* pg = part + g * gstride;
      if (e == 0) {
        pg[0] = m;
        pg[1] = acc;
      } else {
        pg[3 + e] = acc;
      }
    }
  }
  // the last CTA to run out of items puts the work counter back to 0 for the next launch
  __syncthreads();
  if (tid == 0) {
    unsigned int* done = const_cast<unsigned int*>(&wh->done_ctas);
    if (atomicAdd(done, 1u) == gridDim.x - 1) {
      atomicExch(next_item, 0u);
      atomicExch(done, 0u);
    }
  }
}

}  // namespace cobra
