/*
 * cobra.h - C ABI of the KV-COBRA hot path on GB300 (sm_103a).
 *
 * KV-COBRA (arXiv 2609.24298) compresses each attention head's K/V cache by projecting
 * every token onto a per-head, Hadamard-fused, rank-r_h basis and storing b_h-bit codes of
 * a static scalar quantizer (Table alg:kvrobin); decode attention then reads the packed
 * codes directly (Table alg:kvrobin step 8; App. G).
 *
 * Conventions
 *   - Every call returns cobra_status (0 = COBRA_OK); nothing else crosses the ABI.
 *   - The caller owns all memory.  The library never allocates device memory; buffers whose
 *     size depends on the problem have a *_size / *_bytes query.
 *   - "device" pointers are CUDA global-memory addresses on the current device; "host"
 *     pointers are ordinary CPU memory.  `stream` is a cudaStream_t passed as void*
 *     (NULL = the legacy default stream).  Device calls are asynchronous on that stream;
 *     host arrays passed to them are read before the call returns.
 *   - Host-side argument checks run before any launch; a failed check launches nothing.
 *   - Head dimension d is 128 for every device call.
 *   - Device-side waits are bounded; an expired wait is recorded in a device status word
 *     that cobra_check() returns (COBRA_ETIMEOUT) and clears.
 *
 * Packed cache format v1 (the paper fixes only "packed b-bit codes" with no per-token
 * metadata; the bit order is this library's):
 *   code row   128 tokens of one head, 16*r*b bytes.  Strip s = channels (2s, 2s+1),
 *              bytes [32*b*s, 32*b*(s+1)).  Piece p (0..7) of a strip = bytes
 *              [4*b*p, 4*b*(p+1)), b little-endian 32-bit words; word w holds bits
 *              [16w, 16w+16) of sub-stream 0 in its low half and of sub-stream 1 in its high
 *              half; code (rho, h) sits at bits [rho*b, rho*b+b) of sub-stream h, LSB first.
 *   K rows     token t, channel i: piece = (t%16)%8, rho = 2*(t/16) + (t%16)/8, h = i%2.
 *   V rows     token t, channel i: piece = 4*(i%2) + ((t%16)/2)%4, rho = 2*(t/16) + (t%16)/8,
 *              h = (t%16)%2.
 *   regions    head regions start at 256-byte aligned offsets; slot k of a head is at
 *              region + k*16*r*b.  Contiguous: slot = seq*rows_per_seq + row.  Paged
 *              (256-token pages): slot = 2*page_table[seq*pages_per_seq + row/2] + row%2.
 *   tail       codes of tokens past a sequence's length are zero bits; a fresh cache must be
 *              zero-filled before the first cobra_append.
 */
#ifndef COBRA_H
#define COBRA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define COBRA_VERSION 1
#define COBRA_HEAD_DIM 128

typedef enum {
  COBRA_OK = 0,
  COBRA_EINVAL = 1,   /* bad argument: null pointer, size or index out of range, bad shape */
  COBRA_EALIGN = 2,   /* a pointer or offset is not aligned as documented */
  COBRA_EBUDGET = 3,  /* the allocation problem has no feasible solution */
  COBRA_ECUDA = 4,    /* a CUDA runtime call or kernel launch failed */
  COBRA_ETIMEOUT = 5, /* a bounded device-side wait expired (from cobra_check) */
  COBRA_ESPACE = 6    /* a caller-provided buffer is too small */
} cobra_status;

/* Library version (COBRA_VERSION) and a static string for a status code. */
int cobra_version(void);
const char* cobra_status_string(int status);

/* ---------------------------------------------------------------------------------------
 * Allocation (host).  Paper: Eq. (global) min sum_h D_h(r_h, b_h) s.t. sum_h r_h b_h <= B_tot
 * with D(r, b) = sum_{i>r} w_i + q(b) sum_{i<=r} w_i (Eq. drb-preview), q(b) = 2^{-2b}/12
 * (Eq. q); C1 per-head enumeration (Sec. 3.2, App. B), C2 damped proportional update
 * (Sec. 3.3, App. D Eq. c2-update, 5 rounds, eta = 0.3), exact DP (App. E).
 * ------------------------------------------------------------------------------------- */
typedef enum {
  COBRA_ALLOC_DAMPED = 0,  /* C1 + C2 damped update ("water-filling"); the paper's default */
  COBRA_ALLOC_EXACT = 1,   /* exact separable-knapsack DP over per-head (r, b) choices */
  COBRA_ALLOC_UNIFORM = 2  /* C1 only at B_h = bpd*d for every head (the V-side mode, App. vside) */
} cobra_alloc_mode;

typedef struct {
  int mode;        /* cobra_alloc_mode */
  int rounds;      /* C2 rounds (default 5) */
  double eta;      /* C2 damping (default 0.3) */
  int b_min;       /* smallest bit width (default 1; the paper's runs use 2) */
  int b_max;       /* largest bit width (default 8) */
  int r_step;      /* rank grid step (default 2) */
  int allow_r0;    /* rank 0 (head dropped) allowed (default 1) */
  double B_min;    /* C2 budget floor; negative = default (0 if allow_r0 else r_step*b_min) */
  int complete;    /* spend bits the floor leaves unused, greedily (default 1; not in EXACT) */
} cobra_alloc_opts;

/* Fill `o` with the defaults above. */
void cobra_alloc_opts_default(cobra_alloc_opts* o);

/* w: host [n_heads * d] fp64, row h = head h's weights sorted descending (lambda for the MSE
 * objective, sigma_Q^2 * lambda for attention-KL, Prop. kl-bound).  bpd: target bits per
 * dimension, B_tot = n_heads * d * bpd.  Outputs (host, length n_heads, any may be NULL
 * except r and b): r, b, budget (final C2 budget B_h), dist (D_h(r_h, b_h)); *rate_bits =
 * sum r_h b_h.  Errors: EINVAL (bad sizes/options, d > 4096, non-finite w), EBUDGET (no
 * feasible (r, b) for some head with allow_r0 = 0). */
cobra_status cobra_allocate(int n_heads, int d, const double* w, double bpd, const cobra_alloc_opts* opts,
                            int* r, int* b, double* budget, double* dist, long long* rate_bits);

/* Table alg:kvrobin steps 1-2 on the device for many heads at once (one CTA per head, fp64):
 * the same quantities as cobra_calibrate_head - mean, centred (1/N) covariance, its
 * eigen-decomposition (parallel cyclic Jacobi), eigenvalues descending with each
 * eigenvector's largest-magnitude component positive, and with calibration queries the
 * attention-KL weights w_i = sigma_Q,i^2 lambda_i and the stable reorder by w descending
 * (without: w = lambda).  Device inputs: x [n_heads][n_tok][128] fp32 calibration vectors;
 * q [n_heads][n_q][128] fp32 queries of each head's group (n_q = 0 and q = NULL for the MSE
 * objective).  Device outputs (fp64): mu, lam, w [n_heads][128]; U [n_heads][128 * 128] with
 * U[h][j * 128 + i] = component i of direction j (allocator order).  One launch, nothing is
 * synchronised.  Errors: EINVAL, EALIGN (4-byte floats, 8-byte doubles), ECUDA. */
cobra_status cobra_calibrate_heads(int n_heads, int n_tok, const float* x, int n_q, const float* q, double* mu,
                                   double* lam, double* U, double* w, void* stream);

/* App. E "Exact DP over measured distortion", the tables (device, asynchronous on `stream`):
 * every head's calibration tokens go through the deployed quantizer once per candidate
 * (r_list[i], b_list[j]) (W = U_r H_r^T with the head's Hadamard signs, Delta = 2 L_b
 * sigma_bar_r / 2^b rounded to fp32 as cobra_fuse_basis stores it, codes, reconstruction)
 * and D[h][i][j] = (1/n_tok) sum_t sum_k omega_k (u_k . (x_t - x^_t))^2 is written in fp64,
 * omega_k = 1 for the MSE objective or sigma_Q,k^2 for attention-KL, so that r = 0 gives
 * sum_k w_k.  Device inputs, per head h and d = 128: x [n_heads][n_tok][d] fp32 tokens; U
 * [n_heads][d*d] fp32, column k = u_k in the allocator's order; lam, w [n_heads][d] fp64
 * eigenvalues and allocator weights in the same order (cobra_calibrate_heads' outputs: w =
 * lambda for MSE, sigma_Q^2 lambda for attention-KL), from which the library takes omega_k =
 * w_k / lambda_k (0 where lambda_k = 0); mu [n_heads][d] fp32; signs [n_heads][d] int8 (+1/-1).
 * coords: device workspace of n_heads * n_tok * d floats (overwritten).  Host lists: r_list
 * (1..65 entries) strictly ascending in [0, 128], b_list (1..16 entries) in [1, 8].  Two
 * launches; nothing is synchronised.  Errors: EINVAL, EALIGN (4-byte floats, 8-byte
 * doubles), ECUDA. */
cobra_status cobra_measure_distortion(int n_heads, int n_tok, const float* x, const float* U, const double* lam,
                                      const double* w, const float* mu, const int8_t* signs, int n_r,
                                      const int* r_list, int n_b, const int* b_list, float* coords, double* D,
                                      void* stream);

/* App. E "Exact DP over measured distortion": the exact DP of COBRA_ALLOC_EXACT run on
 * explicit per-head distortion tables (e.g. from cobra_measure_distortion) instead of the
 * surrogate.  D: host [n_heads][n_r][n_b] fp64, D[h][i][j] = head h's distortion at
 * (r_list[i], b_list[j]); a row with r_list[i] = 0 means no codes (only its first entry is
 * read).  r_list strictly ascending in [0, d], b_list strictly ascending in [1, 16].
 * Minimises sum_h D_h subject to sum_h r_h b_h <= n_heads * d * bpd; per head and rate the
 * smallest D is kept (the first in (r, b) order on ties), the final pick is the smallest
 * total, then the fewest bits.  Outputs as cobra_allocate (dist may be NULL).  Errors:
 * EINVAL (bad sizes, unsorted lists, non-finite D), EBUDGET (no feasible choice). */
cobra_status cobra_allocate_tables(int n_heads, int d, int n_r, const int* r_list, int n_b, const int* b_list,
                                   const double* D, double bpd, int* r_out, int* b_out, double* dist,
                                   long long* rate_bits);

/* ---------------------------------------------------------------------------------------
 * Calibration helpers (host, fp64).  Table alg:kvrobin steps 1, 2, 5, 6.
 * ------------------------------------------------------------------------------------- */

/* MSE-optimal loading factor L_b of the 2^b-cell clamped uniform quantizer for N(0, 1)
 * (App. A.1 leaves L open; it fixes Delta = 2 L sigma / 2^b).  b in 1..8. */
cobra_status cobra_loading_factor(int b, double* L);

/* H_r (host [r*r] row-major, fp64): normalised Sylvester blocks for the binary digits of r
 * (largest first) times diag(signs[0..r-1]) (Sec. 3.4; equals the scaled Walsh-Hadamard
 * matrix with its sign flip when r is a power of two).  signs: host int8 +1/-1. */
cobra_status cobra_hadamard(int r, const int8_t* signs, double* H);

/* Steps 1-2 for one head.  x: host [n * d] fp32 calibration vectors (row-major).  q: host
 * [nq * d] fp32 calibration queries pooled over the query heads of the group, or NULL for
 * the MSE objective.  Outputs (host): mu [d]; lam [d]; U [d*d] column-major (column j is
 * basis direction j, U[i + j*d]); w [d].  Directions are eigen-ordered (lam descending) for
 * MSE, or reordered by w = sigma_Q^2 lam descending (stable) for KL; each direction's
 * largest-magnitude component is positive.  Covariance is the 1/n centred covariance. */
cobra_status cobra_calibrate_head(int n, int d, const float* x, int nq, const float* q,
                                  double* mu, double* lam, double* U, double* w);

/* Steps 5-6: W = U_r H_r^T (host [d*r] fp32, column-major: W[i + j*d]) and
 * Delta = 2 L_b sigma / 2^b with sigma^2 = mean(lam[0..r-1]).  r = 0 writes nothing and
 * Delta = 0. */
cobra_status cobra_fuse_basis(int d, int r, int b, const double* U, const double* lam, const int8_t* signs,
                              float* W, float* delta);

/* ---------------------------------------------------------------------------------------
 * Layout (host).
 * ------------------------------------------------------------------------------------- */

/* Bytes of one 128-token code row: 16*r*b. */
size_t cobra_row_bytes(int r, int b);

/* 256-byte aligned region offsets (host out [n_heads]) of heads that each hold n_slots rows,
 * heads in index order, and the total cache size in bytes. */
cobra_status cobra_plan_layout(int n_heads, const int* r, const int* b, long long n_slots,
                               uint64_t* head_offsets, uint64_t* total_bytes);

/* ---------------------------------------------------------------------------------------
 * Device parameter block: per-head r, b, Delta, cache offset, fused basis W and mean mu.
 * ------------------------------------------------------------------------------------- */

/* Bytes needed for a parameter block of n_heads heads with ranks r (host [n_heads]). */
cobra_status cobra_params_bytes(int n_heads, const int* r, size_t* bytes);

/* Build the block in caller-allocated device memory `dev_block` (256-byte aligned,
 * `block_bytes` from cobra_params_bytes).  Host inputs: r, b, delta [n_heads]; cache_off
 * [n_heads] (from cobra_plan_layout); W_all = the heads' W (d x r_h column-major) concatenated
 * in head order; mu_all [n_heads * d].  Copies with cudaMemcpyAsync on `stream` from a
 * temporary host image (the call synchronises the stream before returning). */
cobra_status cobra_params_build(void* dev_block, size_t block_bytes, int n_heads, const int* r, const int* b,
                                const float* delta, const uint64_t* cache_off, const float* W_all,
                                const float* mu_all, void* stream);

/* The same block built in host memory (`image`, >= cobra_params_bytes bytes; same inputs as
 * cobra_params_build): the bytes the device block holds, with an FNV-1a 64 checksum in the
 * header.  This is the checkpoint of a calibration (Table alg:kvrobin step 6 stores it once
 * per model): write it to a file, read it back, and upload it with cobra_params_upload. */
cobra_status cobra_params_image(void* image, size_t image_bytes, int n_heads, const int* r, const int* b,
                                const float* delta, const uint64_t* cache_off, const float* W_all,
                                const float* mu_all);

/* Check a host image: magic, version, sizes (image_bytes must equal the block's size), every
 * head's fields and offsets, and the checksum.  COBRA_OK, else COBRA_EINVAL. */
cobra_status cobra_params_verify(const void* image, size_t image_bytes);

/* Verify a host image, then copy it into caller-allocated device memory (256-byte aligned,
 * >= image_bytes) with cudaMemcpyAsync on `stream`; the call synchronises the stream. */
cobra_status cobra_params_upload(void* dev_block, size_t block_bytes, const void* image, size_t image_bytes,
                                 void* stream);

/* ---------------------------------------------------------------------------------------
 * Compression (device).  Table alg:kvrobin step 7: z_t = quantize(W^T (x_t - mu), b*) with
 * the projection and Hadamard as one multiply (Sec. 3.4), packed into the cache (step 8).
 * ------------------------------------------------------------------------------------- */
typedef struct {
  int head0;          /* params index of (layer 0, kv-head 0) of the side being written */
  int layer_stride;   /* params heads between consecutive layers (usually n_kv_heads) */
  int n_layers;       /* layers covered */
  int n_kv_heads;     /* kv heads per layer */
  int side;           /* 0: K rows, 1: V rows (they differ in bit order, see header) */
  int n_seqs;
  int rows_per_seq;   /* contiguous cache: rows (slots) per sequence */
  int pages_per_seq;  /* paged cache: page_table row length (used when page_table != NULL) */
  long long x_stride_layer, x_stride_seq, x_stride_tok, x_stride_head; /* bf16 elements */
} cobra_compress_desc;

/* Compress tokens [t0, t0 + n_tok) of every sequence (t0 a multiple of 128) for every
 * (layer, kv-head) in desc: x (device bf16) at x[l*sl + s*ss + t*st + h*sh + k], k < 128,
 * t counted from t0.  Writes whole code rows (tokens past t0 + n_tok of the last row become
 * zero bits).  cache: device, 256-byte aligned.  page_table: device int32
 * [n_seqs * pages_per_seq] or NULL.  Errors: EINVAL (shapes, t0 % 128 != 0, rows out of
 * range), EALIGN (x not 16-byte aligned or strides not multiples of 8), ECUDA. */
cobra_status cobra_compress(const void* params, const cobra_compress_desc* desc, const void* x, int t0, int n_tok,
                            uint8_t* cache, const int* page_table, void* stream);

/* Append one token per sequence at device position pos[s] (Table alg:kvrobin step 7 applied
 * to the newly decoded token): x at x[l*sl + s*ss + h*sh + k] (x_stride_tok unused).  The
 * token's code bits in its row are replaced (cleared, then set, with atomic word operations);
 * the other tokens' bits are kept.  Appends of different positions of the same row may run
 * concurrently.  A position outside the cache's capacity is skipped and flagged in the device
 * status word (cobra_check returns COBRA_EINVAL). */
cobra_status cobra_append(const void* params, const cobra_compress_desc* desc, const void* x, const int* pos,
                          uint8_t* cache, const int* page_table, void* stream);

/* ---------------------------------------------------------------------------------------
 * Decode attention (device).  Table alg:kvrobin step 8 ("dequantize on attention read") and
 * App. G (dequantisation and inverse rotation in one pass): for every sequence s, layer l,
 * kv head h and query head g of its group,
 *   o = mu_V + W_V Delta_V (sum_t p_t c^V_t / sum_t p_t - (2^{b_V-1} - 1/2)),
 *   p_t = softmax_t(q . K^_t / sqrt(d)),  K^_t = mu_K + W_K Delta_K (c^K_t - 2^{b_K-1} + 1/2),
 * evaluated in rank space over the packed codes (split over token chunks, then combined).
 * ------------------------------------------------------------------------------------- */
typedef struct {
  int k_head0, v_head0; /* params index of (layer 0, kv-head 0) for K and for V */
  int layer_stride;     /* params heads between consecutive layers */
  int n_layers, n_kv_heads;
  int group;            /* query heads per kv head: 4 or 8 */
  int n_seqs;
  int rows_per_seq;     /* contiguous cache */
  int pages_per_seq;    /* paged cache (page_table != NULL) */
  long long q_stride_layer, q_stride_seq; /* bf16 elements; query head j at +j*128 */
  long long o_stride_layer, o_stride_seq; /* fp32 elements; query head j at +j*128 */
} cobra_decode_desc;

/* Workspace bytes for a decode over sequences of at most seq_cap[s] tokens (host [n_seqs]);
 * head_r / head_b: host [>= max params index used] ranks and bit widths of the params. */
cobra_status cobra_decode_workspace_size(const cobra_decode_desc* desc, const int* head_r, const int* head_b,
                                         const int* seq_cap, size_t* bytes);

/* What a plan holds, returned to the host by cobra_decode_plan and passed back to
 * cobra_decode_attn (grid sizes and shared-memory staging need it before launch). */
typedef struct {
  int n_groups;       /* (seq, layer, kv-head) triples */
  int n_items;        /* token chunks */
  int max_row_bytes;  /* largest K or V code row among the planned heads */
  int max_stage_bytes; /* largest K row in whole 16-channel tiles plus V row (128-byte aligned)
                          of a group, for the RoPE decode's staging (0: not known) */
} cobra_decode_info;

/* Write the work plan (token chunks of whole code rows per (seq, layer, kv-head), in the order
 * the scan takes them; the chunks shrink towards the end of the order, so that the scan's warps
 * finish close together) into the
 * device workspace (one cudaMemcpyAsync on `stream`; the call synchronises the stream
 * before returning) and describe it in *info.  The plan stays valid for any
 * seq_lens[s] <= seq_cap[s] and for any parameter block whose heads have the same (r, b). */
cobra_status cobra_decode_plan(const cobra_decode_desc* desc, const int* head_r, const int* head_b, const int* seq_cap,
                               void* workspace, size_t ws_bytes, cobra_decode_info* info, void* stream);

/* The same plan written to host memory instead: `image` receives the first *written bytes of a
 * planned workspace (header, chunk groups, chunks in the order the scan takes them, head-group
 * table); copying them to the start of a workspace of cobra_decode_workspace_size bytes plans
 * it.  With image == NULL (or too small) only *written is set, and the call returns
 * COBRA_EINVAL (COBRA_ESPACE).  Needs no device. */
cobra_status cobra_decode_plan_host(const cobra_decode_desc* desc, const int* head_r, const int* head_b,
                                    const int* seq_cap, void* image, size_t image_bytes, size_t* written,
                                    cobra_decode_info* info);

/* Run decode attention with a planned workspace.  q: device bf16; seq_lens: device int32
 * [n_seqs] (0 gives an all-zero output for that sequence); out: device fp32.  Three
 * launches: query projection, chunked rank-space scan, combine + back-projection.  A head
 * whose code row is larger than info->max_row_bytes is not read; its chunk is marked in the
 * device status word (cobra_check returns COBRA_EINVAL). */
cobra_status cobra_decode_attn(const void* params, const cobra_decode_desc* desc, const cobra_decode_info* info,
                               const void* q, const uint8_t* cache, const int* seq_lens, const int* page_table,
                               float* out, void* workspace, size_t ws_bytes, void* stream);

/* The three stages of cobra_decode_attn as separate calls, in this order on one stream
 * (for callers that overlap them with other work or time them separately):
 *   qproj   q~ = (Delta_K / sqrt d) W_K^T q per (seq, layer, kv-head) into the workspace;
 *   scan    the chunked rank-space pass over the packed codes (online softmax, values in rank
 *           space) writing per-chunk partials into the workspace;
 *   combine merge of the chunks and back-projection o = mu_V + W_V Delta_V (...) into out. */
cobra_status cobra_decode_qproj(const void* params, const cobra_decode_desc* desc, const cobra_decode_info* info,
                                const void* q, void* workspace, size_t ws_bytes, void* stream);
cobra_status cobra_decode_scan(const void* params, const cobra_decode_desc* desc, const cobra_decode_info* info,
                               const uint8_t* cache, const int* seq_lens, const int* page_table, void* workspace,
                               size_t ws_bytes, void* stream);
cobra_status cobra_decode_combine(const void* params, const cobra_decode_desc* desc, const cobra_decode_info* info,
                                  const int* seq_lens, float* out, void* workspace, size_t ws_bytes, void* stream);

/* The query projection fused with the K-side append of Table alg:kvrobin step 7 for one new
 * token per sequence (both project through W_K): kdesc describes the K heads of `desc`
 * (side 0, same head0 = desc->k_head0, layer_stride, n_layers, n_kv_heads and n_seqs, else
 * COBRA_EINVAL); k_new, pos, cache and page_table as for cobra_append.  One launch. */
cobra_status cobra_decode_qproj_append(const void* params, const cobra_decode_desc* desc, const cobra_decode_info* info,
                                       const void* q, const cobra_compress_desc* kdesc, const void* k_new,
                                       const int* pos, uint8_t* cache, const int* page_table, void* workspace,
                                       size_t ws_bytes, void* stream);

/* One decode step: append the new token's K and V codes of every (layer, kv-head, sequence)
 * at pos[s] (Table alg:kvrobin step 7), then decode attention over seq_lens[s] tokens (which
 * normally include the appended one).  kdesc / vdesc describe the K / V heads of `desc`
 * (sides 0 / 1, head0 = desc->k_head0 / desc->v_head0, the other counts equal, else
 * COBRA_EINVAL).  Three launches on `stream`: the query projection with both appends (its
 * grid carries one CTA per (layer, kv head) for the projection and K append, and one for the
 * V append), the scan, the combine; nothing is synchronised.  k_new, v_new, q and out may live in pinned host
 * memory (any memory the device can address): the kernels then read and write it in place. */
cobra_status cobra_decode_step(const void* params, const cobra_decode_desc* desc, const cobra_decode_info* info,
                               const cobra_compress_desc* kdesc, const cobra_compress_desc* vdesc, const void* k_new,
                               const void* v_new, const int* pos, const void* q, uint8_t* cache, const int* seq_lens,
                               const int* page_table, float* out, void* workspace, size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------------------
 * Decode attention for models with the rotary position embedding (RoPE).  Sec. 5 ("Scope")
 * and App. "Post-RoPE experiments": K is compressed before the rotation, so the model's
 * attention turns every reconstructed key to its own position and the query to its position:
 *   p_t = softmax_t(R(p_s) q . R(t) K^_t / sqrt(d)),  o = sum_t p_t V^_t   (V is not rotated),
 * R(x) turning channel pair (j, j + 64) by the angle x * theta^(-2j/128) (the rotate-half
 * form of Llama-3, Mistral and Qwen), key t of a sequence at position t.  The keys are rebuilt
 * from their codes in the 128-dimensional space on the tensor cores (the rotation differs per
 * token, so they cannot be folded into one projected query as cobra_decode_attn does).
 * ------------------------------------------------------------------------------------- */

/* Bytes of the angle table for positions 0 .. max_pos - 1 (1 <= max_pos <= 2^22, else
 * COBRA_EINVAL): 128 floats per position multiple of 16, plus 16 rows for positions 0..15. */
cobra_status cobra_rope_table_bytes(int max_pos, size_t* bytes);

/* Fill the angle table (device, 16-byte aligned, >= cobra_rope_table_bytes) for base theta
 * (> 0; 500000 for Llama-3): cos and sin of x * theta^(-2j/128) evaluated in fp64 and rounded
 * to fp32, for x = 0..15 and x = 16 m.  One launch on `stream`. */
cobra_status cobra_rope_table(double theta, int max_pos, float* table, size_t table_bytes, void* stream);

/* RoPE decode attention with a planned workspace (cobra_decode_plan; the plan and the
 * workspace are the same as for cobra_decode_attn).  q: device bf16; q_pos: device int32
 * [n_seqs] query positions, or NULL for seq_lens[s] - 1; rope_table / max_pos: a table from
 * cobra_rope_table.  A query position or sequence length outside the table, or a head whose
 * code rows do not fit the kernel's staging, is reported through the device status word
 * (cobra_check returns COBRA_EINVAL) and computed with clamped angles or skipped.  The
 * reconstructed keys must stay below 2^14 Delta_K (|mu_K| small against Delta_K 2^15).
 * Three launches: query rotation, scan, combine + back-projection; nothing is synchronised. */
cobra_status cobra_decode_rope_attn(const void* params, const cobra_decode_desc* desc, const cobra_decode_info* info,
                                    const void* q, const int* q_pos, const float* rope_table, int max_pos,
                                    const uint8_t* cache, const int* seq_lens, const int* page_table, float* out,
                                    void* workspace, size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------------------
 * Decode attention without any device allocation.  (The paper has no counterpart; this is an
 * interface convenience.)
 *
 * For callers that cannot allocate device memory - code running where cudaMalloc is not
 * allowed or not wanted, such as an allocator's own callbacks, a process whose memory pool is
 * fixed at start-up, or a plugin that must not touch the device heap - and so cannot provide
 * the workspace cobra_decode_attn needs.  This call computes the same outputs, keeping its
 * workspace in a fixed array of COBRA_STATIC_SCRATCH_BYTES bytes built into the library (it
 * occupies that much memory on every GPU that loads the library, until the process exits).
 *   - No plan or workspace argument: each call plans one token chunk per (seq, layer, kv
 *     head) over the cache's capacity (rows_per_seq, or 2 * pages_per_seq rows when paged)
 *     and writes that plan into the array itself, so nothing has to be zeroed beforehand.
 *   - Returns COBRA_ESPACE when seqs x layers x kv heads chunks do not fit the array
 *     (about 6.4 KB per chunk for group 4, 8.5 KB for group 8).
 *   - The first call on each device looks up the array's address on that device (with the
 *     device current); make that first call before any stream capture.  The address is
 *     looked up again when the current context on the device changes (after cudaDeviceReset,
 *     or with another context made current), so such a call also comes before any capture.
 *   - A descriptor naming a head the parameter block does not hold is reported by cobra_check
 *     (COBRA_EINVAL); that (seq, layer, kv head) is then computed over no tokens.
 *   - All calls on a device share the one array and it keeps the last call's contents: calls
 *     that can overlap on the GPU (different streams, no ordering between them) race and must
 *     not be issued.
 *   - Calls no cudaMalloc / cudaFree or any other allocating routine. */
#define COBRA_STATIC_SCRATCH_BYTES (8u << 20)
cobra_status cobra_decode_attn_static(const void* params, const cobra_decode_desc* desc, const void* q,
                                      const uint8_t* cache, const int* seq_lens, const int* page_table, float* out,
                                      void* stream);

/* Synchronise `stream`, then return and clear the device status word: COBRA_ETIMEOUT if a
 * bounded device wait expired since the last check, COBRA_EINVAL if a kernel skipped work
 * whose size did not fit its launch, COBRA_ECUDA on a CUDA error, else OK. */
cobra_status cobra_check(void* stream);

/* Self-test of the bounded-wait error path (the paper has no counterpart): one warp waits on a
 * shared-memory barrier that nothing completes, gives up after limit_ns nanoseconds
 * (0 < limit_ns <= 100 ms, else COBRA_EINVAL), records the expiry in the device status word
 * exactly as the library's kernels do, and returns.  The next cobra_check(stream) then returns
 * COBRA_ETIMEOUT and the context stays usable. */
cobra_status cobra_selftest_wait_timeout(unsigned long long limit_ns, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* COBRA_H */
