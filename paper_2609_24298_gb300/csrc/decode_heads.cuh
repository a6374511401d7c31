// Per-head kernels of decode attention (Table alg:kvrobin step 8; App. G): the query
// projection ahead of the scan of decode.cuh (optionally fused with the K-side append of one
// new token, step 7, and carrying the V-side append's CTAs in the same launch) and the
// combine + back-projection after it.
#pragma once

#include "compress.cuh"
#include "decode.cuh"

namespace cobra {

// ---------------------------------------------------------------------------------------
// Per-head kernels: the query projection has one CTA of 256 threads per (layer, kv head),
// looping over the sequences 32 query vectors at a time, with the head's basis staged in
// shared memory once; the combine has one per (layer, kv head) and run of kCombineVP query
// vectors.  The workspace's head-group table gives the group of (head, seq).
// ---------------------------------------------------------------------------------------
constexpr int kHeadThreads = 256;
constexpr int kVecPass = 32;  // query vectors (sequences x G) per pass
constexpr int kWLd = 132;     // padded row stride (floats) of a staged basis: conflict-free row reads
// row stride of the transposed rank-space averages of a combine pass of VP vectors (odd:
// the per-channel writes are conflict-free; the reads are broadcasts)
template <int VP>
__host__ __device__ constexpr int combine_zld() {
  return VP + 1;
}

__host__ __device__ constexpr size_t qproj_smem_bytes() {
  return sizeof(float) * ((size_t)kD * kWLd + (size_t)kVecPass * kD + (size_t)kVecPass * kWLd + kD);
}
static_assert(append_smem_bytes() <= qproj_smem_bytes(), "the V-append CTAs use the projection's shared memory");
static_assert(kWLd == kAppendWLd, "the query projection stages W_K as the append reads it");
constexpr int kWtChunk = 64;  // chunk weights held in shared memory per vector and round
constexpr int kCombineVP = 16;  // query vectors per combine CTA (a head's sequences spread over CTAs)
template <int VP>
__host__ __device__ constexpr size_t combine_smem_bytes() {
  return sizeof(float) * ((size_t)kD * combine_zld<VP>() + kD + (size_t)VP * kWtChunk);
}

// ---------------------------------------------------------------------------------------
// a4: query projection
//   q~_g = (Delta_K / sqrt d) log2(e) W_K^T q_g per query head, scaled by a power of two so
//   that max |q~| of the group lands in [256, 512), split into fp16 hi + lo and laid out as
//   the scan's MMA B fragments; Qsum_g = sum over channels of the fed hi + lo values.
//   With ak.x set, the CTA first appends the new K token of every sequence of its head (a8),
//   which projects through the same staged W_K.  With av.x set, the grid has a second half of
//   CTAs (blockIdx.x >= n_qblocks) that append the new V tokens, one (layer, kv head) each, so
//   that both appends and the projection run in one launch.
// ---------------------------------------------------------------------------------------
static_assert(kAppendThreads == kHeadThreads, "the V append runs in the query projection's CTAs");
template <int G>
__global__ void __launch_bounds__(kHeadThreads) qproj_kernel(DecodeArgs a, CompressArgs ak, CompressArgs av,
                                                             int n_qblocks) {
  grid_dep_launch();
  if ((int)blockIdx.x >= n_qblocks) {
    extern __shared__ __align__(16) float vsm[];
    append_block(av, (int)blockIdx.x - n_qblocks, vsm);
    return;
  }
  constexpr int NTK = Heads<G>::NTK, SPP = kVecPass / G;
  extern __shared__ __align__(16) float qsm[];
  float* Ws = qsm;                  // [kD][kWLd]   W_K row i = channel i
  float* Qs = Ws + kD * kWLd;       // [kVecPass][kD] queries of this pass (fp32); the appended tokens first
  float* Os = Qs + kVecPass * kD;   // [kVecPass][kWLd] scaled q~ of this pass
  float* wmu = Os + kVecPass * kWLd;  // [kD] W_K^T mu_K for the append
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
  // the basis is a parameter: its copy overlaps the end of the kernel ahead; the queries, the
  // new tokens, the cache and the q~ blocks of the workspace are touched only after the wait
  const bool append = ak.x != nullptr && r > 0;
  if (append && tid < (r + 3) / 4) cp_async16(smem_addr(wmu + 4 * tid), pool + hk.wmu_off + 4 * tid);
  stage_basis_issue(pool + hk.w_off, r, kWLd, Ws);
  grid_dep_wait();
  if (append) {
    const AppendNext nx = append_load(ak, layer, kv, warp);
    cp_async_wait_all();
    __syncthreads();
    append_tokens(ak, hk, layer, kv, Ws, wmu, Qs + warp * kD, warp, kHeadThreads / 32, nx);
  }
  cp_async_wait_all();
  for (int s0 = 0; s0 < S; s0 += SPP) {
    const int ns = min(SPP, S - s0), nv = ns * G;
    __syncthreads();  // basis staged; the appends and the previous pass are done with Qs and Os
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
        frag[(kap * NTK + nt) * 32 + fl] = make_uint2(pack_f16(e4[0], e4[1]), pack_f16(e4[2], e4[3]));
      }
    }
  }
}

// ---------------------------------------------------------------------------------------
// a7: combine chunks + back-projection
//   per query head: m* = max over chunks, l* = sum 2^(m - m*) l, zbar = Delta_V (sum 2^(m - m*)
//   acc / l* - 2^{b-1} + 1/2), o = mu_V + W_V zbar (zeros for an empty sequence).
// ---------------------------------------------------------------------------------------
// One CTA per (layer, kv head) and run of VP / G sequences (VP query vectors).
template <int G, int VP>
__global__ void __launch_bounds__(kHeadThreads, 4) combine_kernel(DecodeArgs a) {
  constexpr int SPP = VP / G > 0 ? VP / G : 1;
  static_assert(VP % 8 == 0, "combine pass width");
  constexpr int kZLd = combine_zld<VP>();
  extern __shared__ __align__(16) float csm[];
  float* Zs = csm;                  // [kD][kZLd]   zbar of this pass, [channel][vector]
  float* mus = Zs + kD * kZLd;      // [kD]         mu_V
  float* wts = mus + kD;            // [VP][kWtChunk] normalised chunk weights
  __shared__ float vinfo_m[VP], vinfo_inv_l[VP];
  __shared__ int vinfo_first[VP], vinfo_n[VP], vinfo_g[VP], vinfo_seq[VP];
  const WsHeader* wh = reinterpret_cast<const WsHeader*>(a.ws);
  const WsGroup* groups = reinterpret_cast<const WsGroup*>(a.ws + wh->groups_off);
  const float* parts = reinterpret_cast<const float*>(a.ws + wh->part_off);
  const int S = wh->n_seqs;
  const int nchunks = (S + SPP - 1) / SPP;
  const int chunk = blockIdx.x % nchunks;
  const int* hg = reinterpret_cast<const int*>(a.ws + wh->hg_off) + (size_t)(blockIdx.x / nchunks) * S;
  const WsGroup g0 = groups[hg[0]];
  const HeadEntry hv = head_table(a.block)[g0.v_head];
  const float* pool = param_pool(a.block);
  const int rv = hv.r, layer = g0.layer, kv = g0.kv;
  const int tid = threadIdx.x;
  const float cen = rv > 0 ? (float)(1 << (hv.b - 1)) - 0.5f : 0.f;
  if (tid < kD) mus[tid] = pool[hv.mu_off + tid];
  // the rows of W_V are read through L1 in the back-projection (every warp reads the same rows);
  // they are pulled into L2 here, while the scan ahead of this kernel is still finishing
  const float4* W4 = reinterpret_cast<const float4*>(pool + hv.w_off);
  for (int idx = tid; idx < rv * (kD / 32); idx += kHeadThreads) prefetch_l2(pool + hv.w_off + 32 * idx);
  // the plan side of every vector: its group's chunks and query head
  const int s0 = chunk * SPP;
  const int ns = min(SPP, S - s0), nv = ns * G;
  if (tid < nv) {
    const WsGroup gr = groups[hg[s0 + tid / G]];
    vinfo_first[tid] = gr.first_item;
    vinfo_n[tid] = gr.n_items;
    vinfo_g[tid] = tid % G;
    vinfo_seq[tid] = gr.seq;
  }
  // the appends of the next step may start their parameter staging meanwhile
  grid_dep_launch();
  // everything above is independent of the scan; its partials are read only from here on
  grid_dep_wait();
  {
    __syncthreads();  // mu_V and the vector table staged
    // (1) per vector (warp w: vectors w, w + 8, ...): m* = max over the chunks and
    //     l* = sum 2^(m - m*) l, lanes over chunks, merged online (a chunk with no tokens has
    //     m = -inf and no value entries; its weight is zero).  The vectors' loads are issued
    //     together; the lanes keep the m of the first kWtChunk chunks and turn them into the
    //     weights 2^(m - m*) / l* of the first round of (2).
    const int warp = tid >> 5, lane = tid & 31;
    constexpr int NU = VP / (kHeadThreads / 32);
    {
      const float* pg0[NU];
      int ni[NU];
      float M[NU], Lsum[NU];
      int kmax = 0;
#pragma unroll
      for (int u = 0; u < NU; ++u) {
        const int v = warp + 8 * u;
        ni[u] = (v < nv && a.seq_lens[vinfo_seq[v]] > 0) ? vinfo_n[v] : 0;
        pg0[u] = parts + (v < nv ? (size_t)vinfo_first[v] * wh->part_stride + (v % G) * wh->g_stride : 0);
        M[u] = -INFINITY;
        Lsum[u] = 0.f;
        kmax = max(kmax, ni[u]);
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
          if (k < kWtChunk && warp + 8 * u < nv) wts[(warp + 8 * u) * kWtChunk + k] = mk[u];
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
        if (v >= nv) continue;
        const float inv_l = ni[u] > 0 ? 1.f / Lsum[u] : 0.f;
        if (lane == 0) {
          vinfo_first[v] = ni[u] > 0 ? vinfo_first[v] : -1;
          vinfo_n[v] = ni[u];
          vinfo_m[v] = M[u];
          vinfo_inv_l[v] = inv_l;
        }
        // the same lane wrote wts[v][k] above for k < kmax
        for (int k = lane; k < kWtChunk; k += 32) {
          const float mk = k < ni[u] ? wts[v * kWtChunk + k] : -INFINITY;
          wts[v * kWtChunk + k] = mk != -INFINITY ? exp2f(mk - M[u]) * inv_l : 0.f;
        }
      }
    }
    __syncthreads();
    // (2) zbar[v][i] = Delta (sum_k w_k acc_k[i] - 2^{b-1} + 1/2) with w_k = 2^(m_k - m*) / l*.
    //     Rounds of kWtChunk chunks (the first round's weights come from (1); later rounds
    //     compute them one (vector, chunk) per thread into shared memory).  Thread (channel
    //     quad cq, slot) of rw = r_V rounded up to 32, 64 or 128 channels holds channels
    //     4 cq .. 4 cq + 3 of the vectors slot, slot + ns, ... (ns = 256 / (rw / 4) slots) and
    //     sums over the chunks in blocks of KB, the 16-byte loads of all its vectors' KB chunks
    //     issued before any is used.
    {
      constexpr int VPT = (VP + 7) / 8;  // vectors per thread at most (ns >= 8)
      constexpr int KB = VPT >= 4 ? 4 : 8;  // chunks per block: VPT x KB 16-byte loads in flight
      const int rw = rv <= 32 ? 32 : rv <= 64 ? 64 : kD;
      const int nq = rw / 4, ns = kHeadThreads / nq;
      const int cq = tid % nq, slot = tid / nq;
      const int pstride = wh->part_stride;
      int kmax = 0;
      for (int v = 0; v < nv; ++v) kmax = max(kmax, vinfo_n[v]);
      float4 acc[VPT];
#pragma unroll
      for (int q = 0; q < VPT; ++q) acc[q] = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int k0 = 0; k0 < kmax; k0 += kWtChunk) {
        if (k0 > 0) {
          __syncthreads();  // the previous round's weights are consumed
          for (int idx = tid; idx < nv * kWtChunk; idx += kHeadThreads) {
            const int v = idx / kWtChunk, k = k0 + idx % kWtChunk;
            float w = 0.f;
            if (k < vinfo_n[v]) {
              const float mk = parts[(size_t)(vinfo_first[v] + k) * pstride + vinfo_g[v] * wh->g_stride];
              if (mk != -INFINITY) w = exp2f(mk - vinfo_m[v]) * vinfo_inv_l[v];
            }
            wts[idx] = w;
          }
          __syncthreads();
        }
        if (4 * cq >= rv) continue;
        const int kr = min(kWtChunk, kmax - k0);
        for (int kb = 0; kb < kr; kb += KB) {
          float4 x[VPT][KB];
#pragma unroll
          for (int q = 0; q < VPT; ++q) {
            const int v = slot + ns * q;
            const int n = v < nv ? vinfo_n[v] - k0 : 0;
            // the partial's channels start 4 floats in and every stride is a multiple of 4 floats
            const float4* px = reinterpret_cast<const float4*>(
                parts + (size_t)max(vinfo_first[v < nv ? v : 0], 0) * pstride + (size_t)k0 * pstride +
                (v < nv ? vinfo_g[v] : 0) * wh->g_stride + 4 + 4 * cq);
#pragma unroll
            for (int kk = 0; kk < KB; ++kk)
              x[q][kk] = (kb + kk < n) ? px[(size_t)(kb + kk) * (pstride / 4)] : make_float4(0.f, 0.f, 0.f, 0.f);
          }
#pragma unroll
          for (int q = 0; q < VPT; ++q) {
            const int v = slot + ns * q;
            if (v >= nv) break;
            const float* wv = wts + v * kWtChunk + kb;
#pragma unroll
            for (int kk = 0; kk < KB; ++kk) {
              const float w = (kb + kk < kWtChunk) ? wv[kk] : 0.f;
              if (w != 0.f) {  // an empty chunk's value entries were never written
                acc[q].x += w * x[q][kk].x;
                acc[q].y += w * x[q][kk].y;
                acc[q].z += w * x[q][kk].z;
                acc[q].w += w * x[q][kk].w;
              }
            }
          }
        }
      }
      if (4 * cq < rv) {
#pragma unroll
        for (int q = 0; q < VPT; ++q) {
          const int v = slot + ns * q;
          if (v >= nv) break;
          const bool live = vinfo_first[v] >= 0;
          const float a4[4] = {acc[q].x, acc[q].y, acc[q].z, acc[q].w};
#pragma unroll
          for (int c = 0; c < 4; ++c)
            if (4 * cq + c < rv) Zs[(4 * cq + c) * kZLd + v] = live ? hv.delta * (a4[c] - cen) : 0.f;
        }
      }
    }
    __syncthreads();
    // thread: dims 4 (tid % 32) .. +3 for vectors VPW (tid / 32) .. +VPW-1
    constexpr int VPW = VP / (kHeadThreads / 32);
    const int d0 = 4 * (tid & 31), v0 = VPW * (tid >> 5);
    if (v0 < nv) {
      const float4 m4 = *reinterpret_cast<const float4*>(mus + d0);
      float4 o[VPW];
#pragma unroll
      for (int v = 0; v < VPW; ++v) o[v] = m4;
      auto accum = [&](const float4& w, int i) {
        float zz[VPW];
#pragma unroll
        for (int v = 0; v < VPW; ++v) zz[v] = Zs[i * kZLd + v0 + v];
#pragma unroll
        for (int v = 0; v < VPW; ++v) {
          o[v].x += w.x * zz[v];
          o[v].y += w.y * zz[v];
          o[v].z += w.z * zz[v];
          o[v].w += w.w * zz[v];
        }
      };
      // rows in blocks of 8 whose loads are all issued before the first is used
      int i = 0;
      for (; i + 8 <= rv; i += 8) {
        float4 w[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) w[u] = __ldg(W4 + (i + u) * (kD / 4) + (d0 >> 2));
#pragma unroll
        for (int u = 0; u < 8; ++u) accum(w[u], i + u);
      }
      for (; i < rv; ++i) accum(__ldg(W4 + i * (kD / 4) + (d0 >> 2)), i);
#pragma unroll
      for (int v = 0; v < VPW; ++v) {
        const int vv = v0 + v;
        if (vv >= nv) break;
        const int seq = s0 + vv / G, g = vv % G;
        const bool empty = vinfo_first[vv] < 0;  // a sequence without tokens
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
