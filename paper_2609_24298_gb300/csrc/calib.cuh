// One-time calibration on the device (Table alg:kvrobin steps 1-2; App. F "Calibration"),
// one CTA per head, fp64 throughout:
//   step 1  mean and centred (1/N) covariance of the head's calibration vectors, symmetric
//           eigen-decomposition by parallel cyclic Jacobi (each round applies 64 disjoint
//           rotations, a round-robin schedule covers every pair once per sweep), eigenvalues
//           descending, each eigenvector's largest-magnitude component made positive;
//   step 2  with calibration queries: sigma_Q,i^2 = mean (u_i . q)^2, weights
//           w_i = sigma_Q,i^2 lambda_i and the basis reordered by w descending (stable);
//           without: w = lambda in eigen order.
// Shared memory: the covariance as its packed upper triangle (A[i][j], i <= j) and the
// eigenvectors V (row-major, column j = eigenvector j); the token tiles of the covariance
// pass reuse V's space before the rotations start.
#pragma once

#include "common.cuh"

namespace cobra {

constexpr int kCalThreads = 256;
constexpr int kCalPairs = kD / 2;             // disjoint rotations per round
constexpr int kCalPacked = kD * (kD + 1) / 2;  // packed upper triangle
constexpr int kCalMaxSweeps = 40;
constexpr int kCalTile = 32;  // tokens per covariance tile
static_assert(kCalThreads == 2 * kD, "two threads per direction and per covariance row");

__host__ __device__ constexpr size_t calib_smem_bytes() {
  return sizeof(double) * ((size_t)kCalPacked + (size_t)kD * kD + 4 * kCalPairs + 2 * kD + kCalThreads);
}

struct CalibArgs {
  const float* x;  // [n_heads][n_tok][kD]
  const float* q;  // [n_heads][n_q][kD] or null
  double* mu;      // [n_heads][kD]
  double* lam;     // [n_heads][kD]  (allocator order)
  double* U;       // [n_heads][kD * kD], column j = direction j (allocator order)
  double* w;       // [n_heads][kD]
  int n_tok, n_q;
};

__device__ __forceinline__ int packed_index(int i, int j) {  // i <= j
  return i * kD - (i * (i - 1)) / 2 + (j - i);
}
__device__ __forceinline__ double packed_get(const double* A, int i, int j) {
  return i <= j ? A[packed_index(i, j)] : A[packed_index(j, i)];
}
// round-robin pairing of round k (0 .. kD-2): pair 0 = (kD-1, k), pair m = ((k+m) mod (kD-1),
// (k-m) mod (kD-1)); every unordered pair appears in exactly one round
__device__ __forceinline__ void rr_pair(int k, int m, int& p, int& q) {
  constexpr int n1 = kD - 1;
  int a, b;
  if (m == 0) {
    a = n1;
    b = k;
  } else {
    a = (k + m) % n1;
    b = (k - m + n1) % n1;
  }
  p = min(a, b);
  q = max(a, b);
}

__device__ double block_sum(double v, double* scratch) {
  const int tid = threadIdx.x;
  scratch[tid] = v;
  __syncthreads();
  for (int s = kCalThreads / 2; s > 0; s >>= 1) {
    if (tid < s) scratch[tid] += scratch[tid + s];
    __syncthreads();
  }
  const double r = scratch[0];
  __syncthreads();
  return r;
}

__global__ void __launch_bounds__(kCalThreads, 1) calib_kernel(CalibArgs a) {
  extern __shared__ __align__(16) double csmem[];
  double* A = csmem;                      // packed upper triangle
  double* V = A + kCalPacked;             // [kD][kD] row-major
  double* rot = V + kD * kD;              // [kCalPairs][4]: c, s, p, q
  double* mu = rot + 4 * kCalPairs;       // [kD]
  double* vals = mu + kD;                 // [kD]
  double* scratch = vals + kD;            // [kCalThreads]
  const int h = blockIdx.x, tid = threadIdx.x;
  const float* x = a.x + (size_t)h * a.n_tok * kD;
  const double inv_n = 1.0 / (double)a.n_tok;

  // ---- step 1: mean, centred covariance (upper triangle), in fp64 ----
  if (tid < kD) {
    double s = 0.0;
    for (int t = 0; t < a.n_tok; ++t) s += (double)x[(size_t)t * kD + tid];
    mu[tid] = s * inv_n;
  }
  __syncthreads();
  double* xt = V;  // token tile [kCalTile][kD], centred
  // thread: row i = tid / 2, columns j in [32 c0, 32 c0 + 32) of pass `pass` for its half
  const int ri = tid >> 1;
  for (int pass = 0; pass < 2; ++pass) {
    const int c0 = 64 * pass + 32 * (tid & 1);
    double acc[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) acc[j] = 0.0;
    for (int t0 = 0; t0 < a.n_tok; t0 += kCalTile) {
      const int nt = min(kCalTile, a.n_tok - t0);
      __syncthreads();
      for (int idx = tid; idx < kCalTile * kD; idx += kCalThreads) {
        const int t = idx / kD, i = idx % kD;
        xt[idx] = t < nt ? (double)x[(size_t)(t0 + t) * kD + i] - mu[i] : 0.0;
      }
      __syncthreads();
      for (int t = 0; t < nt; ++t) {
        const double xi = xt[t * kD + ri];
#pragma unroll
        for (int j = 0; j < 32; ++j) acc[j] = fma(xi, xt[t * kD + c0 + j], acc[j]);
      }
    }
#pragma unroll
    for (int j = 0; j < 32; ++j)
      if (c0 + j >= ri) A[packed_index(ri, c0 + j)] = acc[j] * inv_n;
  }
  __syncthreads();
  // V = I
  for (int idx = tid; idx < kD * kD; idx += kCalThreads) V[idx] = (idx / kD == idx % kD) ? 1.0 : 0.0;
  double scale2 = 0.0;
  for (int e = tid; e < kCalPacked; e += kCalThreads) scale2 += A[e] * A[e];
  const double scale = sqrt(block_sum(scale2, scratch));

  // ---- parallel cyclic Jacobi ----
  for (int sweep = 0; sweep < kCalMaxSweeps; ++sweep) {
    double off = 0.0;
    for (int idx = tid; idx < kD * kD; idx += kCalThreads) {
      const int i = idx / kD, j = idx % kD;
      if (j > i) {
        const double v = A[packed_index(i, j)];
        off += v * v;
      }
    }
    off = block_sum(off, scratch);
    if (off == 0.0 || sqrt(off) <= 1e-15 * scale) break;
    for (int k = 0; k < kD - 1; ++k) {
      if (tid < kCalPairs) {
        int p, q;
        rr_pair(k, tid, p, q);
        const double apq = A[packed_index(p, q)];
        double c = 1.0, s = 0.0;
        if (apq != 0.0) {
          const double app = A[packed_index(p, p)], aqq = A[packed_index(q, q)];
          const double theta = (aqq - app) / (2.0 * apq);
          const double t = (theta >= 0 ? 1.0 : -1.0) / (fabs(theta) + sqrt(theta * theta + 1.0));
          c = 1.0 / sqrt(t * t + 1.0);
          s = t * c;
        }
        rot[4 * tid + 0] = c;
        rot[4 * tid + 1] = s;
        rot[4 * tid + 2] = p;
        rot[4 * tid + 3] = q;
      }
      __syncthreads();
      // A <- J^T A J on every 2x2 block (pair P, pair Q), P <= Q; J maps column p to
      // c e_p - s e_q and column q to s e_p + c e_q
      for (int blk = tid; blk < kCalPairs * kCalPairs; blk += kCalThreads) {
        const int P = blk / kCalPairs, Q = blk % kCalPairs;
        if (Q < P) continue;
        const double c1 = rot[4 * P], s1 = rot[4 * P + 1], c2 = rot[4 * Q], s2 = rot[4 * Q + 1];
        const int p1 = (int)rot[4 * P + 2], q1 = (int)rot[4 * P + 3], p2 = (int)rot[4 * Q + 2], q2 = (int)rot[4 * Q + 3];
        if (P == Q) {
          const double app = A[packed_index(p1, p1)], aqq = A[packed_index(q1, q1)], apq = A[packed_index(p1, q1)];
          // rows and columns p, q of the symmetric 2x2 block
          A[packed_index(p1, p1)] = c1 * c1 * app - 2.0 * s1 * c1 * apq + s1 * s1 * aqq;
          A[packed_index(q1, q1)] = s1 * s1 * app + 2.0 * s1 * c1 * apq + c1 * c1 * aqq;
          A[packed_index(p1, q1)] = 0.0;
        } else {
          const double a11 = packed_get(A, p1, p2), a12 = packed_get(A, p1, q2);
          const double a21 = packed_get(A, q1, p2), a22 = packed_get(A, q1, q2);
          // columns: [a11 a12; a21 a22] J2
          const double b11 = c2 * a11 - s2 * a12, b12 = s2 * a11 + c2 * a12;
          const double b21 = c2 * a21 - s2 * a22, b22 = s2 * a21 + c2 * a22;
          // rows: J1^T [b]
          const double n11 = c1 * b11 - s1 * b21, n21 = s1 * b11 + c1 * b21;
          const double n12 = c1 * b12 - s1 * b22, n22 = s1 * b12 + c1 * b22;
          A[p1 <= p2 ? packed_index(p1, p2) : packed_index(p2, p1)] = n11;
          A[p1 <= q2 ? packed_index(p1, q2) : packed_index(q2, p1)] = n12;
          A[q1 <= p2 ? packed_index(q1, p2) : packed_index(p2, q1)] = n21;
          A[q1 <= q2 ? packed_index(q1, q2) : packed_index(q2, q1)] = n22;
        }
      }
      // V <- V J
      for (int idx = tid; idx < kD * kCalPairs; idx += kCalThreads) {
        const int row = idx / kCalPairs, P = idx % kCalPairs;
        const double c = rot[4 * P], s = rot[4 * P + 1];
        const int p = (int)rot[4 * P + 2], q = (int)rot[4 * P + 3];
        const double vp = V[row * kD + p], vq = V[row * kD + q];
        V[row * kD + p] = c * vp - s * vq;
        V[row * kD + q] = s * vp + c * vq;
      }
      __syncthreads();
    }
  }

  // ---- eigenvalues descending (stable), sign rule, weights, order ----
  if (tid < kD) vals[tid] = A[packed_index(tid, tid)];
  __syncthreads();
  // rank of eigenvalue j in descending order (ties: the lower index first)
  int rank_e = 0;
  if (tid < kD) {
    const double v = vals[tid];
    for (int k = 0; k < kD; ++k) rank_e += (vals[k] > v) || (vals[k] == v && k < tid);
  }
  // sign of eigenvector tid: its largest-magnitude component (first on ties) made positive
  double sgn = 1.0;
  if (tid < kD) {
    double vmax = -1.0, vs = 0.0;
    for (int i = 0; i < kD; ++i) {
      const double vv = V[i * kD + tid];
      if (fabs(vv) > vmax) {
        vmax = fabs(vv);
        vs = vv;
      }
    }
    sgn = vs < 0 ? -1.0 : 1.0;
  }
  // query variance along eigenvector j (fp64), the queries split between two threads per
  // direction; then w
  double wv = 0.0;
  if (a.q) {
    const int j = tid & (kD - 1), half = tid >> 7;
    const float* q = a.q + (size_t)h * a.n_q * kD;
    double acc = 0.0;
    for (int t = half; t < a.n_q; t += 2) {
      double p = 0.0;
      for (int i = 0; i < kD; ++i) p += V[i * kD + j] * (double)q[(size_t)t * kD + i];
      acc += p * p;
    }
    if (half) scratch[j] = acc;
    __syncthreads();
    if (!half) wv = (acc + scratch[j]) / (double)a.n_q * vals[j];
  } else if (tid < kD) {
    wv = vals[tid];
  }
  // final position: the eigen order, then (with queries) a stable sort of -w over it
  __syncthreads();
  double* wsort = scratch;  // [kD] w by eigen rank
  double* vsort = scratch + kD;
  if (tid < kD) {
    wsort[rank_e] = wv;
    vsort[rank_e] = vals[tid];
  }
  __syncthreads();
  int pos = 0;
  if (tid < kD) {
    pos = rank_e;
    if (a.q) {
      pos = 0;
      const double v = wsort[rank_e];
      for (int k = 0; k < kD; ++k) pos += (wsort[k] > v) || (wsort[k] == v && k < rank_e);
    }
    a.lam[(size_t)h * kD + pos] = vals[tid];
    a.w[(size_t)h * kD + pos] = wv;
    double* Uo = a.U + (size_t)h * kD * kD + (size_t)pos * kD;
    for (int i = 0; i < kD; ++i) Uo[i] = sgn * V[i * kD + tid];
    a.mu[(size_t)h * kD + tid] = mu[tid];
  }
}

}  // namespace cobra
