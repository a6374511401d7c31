// libcobra device entry points: argument checks and launches for compress, append and
// decode attention, plus the device status check.
#include <cstddef>
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cstring>

#include "../../include/cobra.h"
#include "common.cuh"
#include "compress.cuh"
#include "compress_tc.cuh"
#include "decode.cuh"
#include "decode_heads.cuh"
#include "measure.cuh"
#include "calib.cuh"
#include "rope.cuh"

using namespace cobra;

namespace {

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

cobra_status launch_status() {
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? COBRA_OK : COBRA_ECUDA;
}

cobra_status check_compress_desc(const cobra_compress_desc* d) {
  if (!d) return COBRA_EINVAL;
  if (d->n_layers < 1 || d->n_kv_heads < 1 || d->n_seqs < 1 || d->head0 < 0 || d->layer_stride < d->n_kv_heads ||
      (d->side != 0 && d->side != 1) || d->rows_per_seq < 0 || d->pages_per_seq < 0)
    return COBRA_EINVAL;
  return COBRA_OK;
}

int sm_count() {
  int dev = 0, n = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  return n > 0 ? n : 1;
}

// The dynamic shared memory a kernel may use is granted per device (cudaFuncSetAttribute acts
// on the current device), so each launch site keeps, per device, the largest size granted.
constexpr int kMaxDevices = 64;
using Granted = std::atomic<size_t>[kMaxDevices];

template <typename Kernel>
cobra_status ensure_smem(Kernel kernel, size_t bytes, Granted& granted) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return COBRA_ECUDA;
  size_t cur = granted[dev].load(std::memory_order_relaxed);
  if (bytes <= cur) return COBRA_OK;
  if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes) != cudaSuccess)
    return COBRA_ECUDA;
  while (bytes > cur && !granted[dev].compare_exchange_weak(cur, bytes)) {
  }
  return COBRA_OK;
}

}  // namespace

namespace {

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_tiled() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// 5-D tensor map over x (bf16): dimension 0 = the 128 head dims (contiguous), the other four
// (kv head, token, sequence, layer) ordered by increasing stride as the TMA unit requires.
// Box: 64 dims x 128 tokens, 128-byte swizzle; tokens past n_tok read as zeros.
cobra_status make_x_map(const cobra_compress_desc* d, const void* x, int n_tok, CUtensorMap* map, int slots[4]) {
  EncodeTiledFn enc = encode_tiled();
  if (!enc) return COBRA_ECUDA;
  struct Dim {
    long long size, stride_bytes;
    int box, logical;
  };
  Dim dims[4] = {{d->n_kv_heads, d->x_stride_head * 2, 1, 0},
                 {n_tok, d->x_stride_tok * 2, kRowTokens, 1},
                 {d->n_seqs, d->x_stride_seq * 2, 1, 2},
                 {d->n_layers, d->x_stride_layer * 2, 1, 3}};
  // a dimension of size 1 is never stepped: give it a stride that keeps the order valid
  long long run = 256;
  for (int pass = 0; pass < 4; ++pass)
    for (auto& e : dims)
      if (e.size > 1) run = std::max(run, e.stride_bytes * e.size);
  for (auto& e : dims)
    if (e.size == 1) e.stride_bytes = run;
  std::stable_sort(dims, dims + 4, [](const Dim& p, const Dim& q) { return p.stride_bytes < q.stride_bytes; });
  cuuint64_t gdim[5] = {(cuuint64_t)kD, 0, 0, 0, 0};
  cuuint64_t gstride[4];
  cuuint32_t box[5] = {64, 1, 1, 1, 1};
  cuuint32_t estride[5] = {1, 1, 1, 1, 1};
  for (int i = 0; i < 4; ++i) {
    if (dims[i].stride_bytes <= 0 || dims[i].stride_bytes % 16 || dims[i].size < 1) return COBRA_EINVAL;
    gdim[i + 1] = (cuuint64_t)dims[i].size;
    gstride[i] = (cuuint64_t)dims[i].stride_bytes;
    box[i + 1] = (cuuint32_t)dims[i].box;
    slots[dims[i].logical] = i + 1;
  }
  const CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void*>(x), gdim, gstride, box, estride,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? COBRA_OK : COBRA_EINVAL;
}

}  // namespace

extern "C" cobra_status cobra_compress(const void* params, const cobra_compress_desc* d, const void* x, int t0, int n_tok,
                                       uint8_t* cache, const int* page_table, void* stream) {
  cobra_status st = check_compress_desc(d);
  if (st != COBRA_OK) return st;
  if (!params || !x || !cache || n_tok < 0 || t0 < 0 || (t0 % kRowTokens) != 0) return COBRA_EINVAL;
  if (!aligned(params, 256) || !aligned(cache, 256) || !aligned(x, 16)) return COBRA_EALIGN;
  if ((d->x_stride_seq % 8) || (d->x_stride_tok % 8) || (d->x_stride_head % 8) || (d->x_stride_layer % 8))
    return COBRA_EALIGN;
  const long long last_row = (t0 + (long long)n_tok + kRowTokens - 1) / kRowTokens;
  if (page_table) {
    if (d->pages_per_seq < 1 || last_row > 2LL * d->pages_per_seq) return COBRA_EINVAL;
  } else if (last_row > d->rows_per_seq) {
    return COBRA_EINVAL;
  }
  if (n_tok == 0) return COBRA_OK;
  CUtensorMap map;
  int slots[4];
  st = make_x_map(d, x, n_tok, &map, slots);
  if (st != COBRA_OK) return st;
  static Granted granted;
  if (ensure_smem(compress_tc_kernel, kTcSmemBytes, granted) != COBRA_OK) return COBRA_ECUDA;
  TcArgs a{};
  a.block = static_cast<const unsigned char*>(params);
  a.cache = cache;
  a.page_table = page_table;
  a.head0 = d->head0;
  a.layer_stride = d->layer_stride;
  a.n_kv = d->n_kv_heads;
  a.side = d->side;
  a.n_seqs = d->n_seqs;
  a.rows_per_seq = d->rows_per_seq;
  a.pages_per_seq = d->pages_per_seq;
  a.t0 = t0;
  a.n_tok = n_tok;
  a.slot_head = slots[0];
  a.slot_tok = slots[1];
  a.slot_seq = slots[2];
  a.slot_layer = slots[3];
  const long long heads = (long long)d->n_layers * d->n_kv_heads;
  const long long tiles = (long long)d->n_seqs * ((n_tok + kRowTokens - 1) / kRowTokens);
  // One CTA per SM at a time.  Split each head's tiles into the number of chunks that fills
  // whole waves of SMs best (the last wave of a ragged grid idles SMs), keeping at least 16
  // tiles per CTA so that converting the head's basis stays a small part of its work.
  const long long sms = sm_count();
  const long long cmax = std::max(1LL, std::min(tiles / 16, 8 * sms));
  long long chunks = 1;
  double best = -1.0;
  for (long long c = 1; c <= cmax; ++c) {
    const long long total = heads * c, waves = (total + sms - 1) / sms;
    const double eff = (double)total / (double)(waves * sms);
    if (eff > best + 1e-9) {
      best = eff;
      chunks = c;
    }
  }
  a.chunks = (int)chunks;
  const long long grid = heads * chunks;
  if (grid > 0x7fffffffLL) return COBRA_EINVAL;
  compress_tc_kernel<<<(unsigned)grid, kTcThreads, kTcSmemBytes, (cudaStream_t)stream>>>(map, a);
  return launch_status();
}

namespace {
// Launch with programmatic stream serialisation: the kernel may become resident while the one
// ahead of it in the stream finishes; it waits for that kernel (grid_dep_wait) before touching
// anything the kernel ahead may produce or read.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), unsigned grid, unsigned block, size_t smem, cudaStream_t s,
                       Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(block);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}
}  // namespace

namespace {
// validated append arguments for one side
cobra_status append_args(const void* params, const cobra_compress_desc* d, const void* x, const int* pos,
                         uint8_t* cache, const int* page_table, CompressArgs& a) {
  cobra_status st = check_compress_desc(d);
  if (st != COBRA_OK) return st;
  if (!params || !x || !pos || !cache) return COBRA_EINVAL;
  if (!aligned(params, 256) || !aligned(cache, 256) || !aligned(x, 2)) return COBRA_EALIGN;
  if (page_table && d->pages_per_seq < 1) return COBRA_EINVAL;
  if ((long long)d->n_layers * d->n_kv_heads > 0x7fffffffLL) return COBRA_EINVAL;
  a = CompressArgs{};
  a.block = static_cast<const unsigned char*>(params);
  a.x = static_cast<const __nv_bfloat16*>(x);
  a.cache = cache;
  a.page_table = page_table;
  a.pos = pos;
  a.sl = d->x_stride_layer;
  a.ss = d->x_stride_seq;
  a.sh = d->x_stride_head;
  a.head0 = d->head0;
  a.layer_stride = d->layer_stride;
  a.n_layers = d->n_layers;
  a.n_kv = d->n_kv_heads;
  a.side = d->side;
  a.n_seqs = d->n_seqs;
  a.rows_per_seq = d->rows_per_seq;
  a.pages_per_seq = d->pages_per_seq;
  return COBRA_OK;
}
}  // namespace

extern "C" cobra_status cobra_append(const void* params, const cobra_compress_desc* d, const void* x, const int* pos,
                                     uint8_t* cache, const int* page_table, void* stream) {
  CompressArgs a;
  cobra_status st = append_args(params, d, x, pos, cache, page_table, a);
  if (st != COBRA_OK) return st;
  const long long grid = (long long)d->n_layers * d->n_kv_heads;  // one CTA per (layer, kv head)
  static Granted granted;
  if (ensure_smem(append_kernel, append_smem_bytes(), granted) != COBRA_OK) return COBRA_ECUDA;
  if (launch_pdl(append_kernel, (unsigned)grid, kAppendThreads, append_smem_bytes(), (cudaStream_t)stream, a) !=
      cudaSuccess)
    return COBRA_ECUDA;
  return launch_status();
}

namespace {

enum Stage { kQproj = 1, kScan = 2, kCombine = 4 };

template <int G>
cobra_status launch_decode(const DecodeArgs& a, int n_heads, int n_seqs, int n_items, int stages, cudaStream_t s,
                           bool after_plan_kernel = false, const CompressArgs& ak = CompressArgs{},
                           const CompressArgs& av = CompressArgs{}) {
  static Granted qproj_granted, combine_granted;
  if (ensure_smem(qproj_kernel<G>, qproj_smem_bytes(), qproj_granted) != COBRA_OK ||
      ensure_smem(combine_kernel<G, kCombineVP>, combine_smem_bytes<kCombineVP>(), combine_granted) != COBRA_OK)
    return COBRA_ECUDA;
  if (stages & kQproj) {
    // the query projection reads the plan before its wait; right after the plan kernel it is
    // launched in plain stream order
    // with a V append, its CTAs follow the projection's (one per (layer, kv head))
    const unsigned grid = (unsigned)n_heads * (av.x ? 2u : 1u);
    if (after_plan_kernel) {
      qproj_kernel<G><<<grid, kHeadThreads, qproj_smem_bytes(), s>>>(a, ak, av, n_heads);
      if (cudaGetLastError() != cudaSuccess) return COBRA_ECUDA;
    } else if (launch_pdl(qproj_kernel<G>, grid, kHeadThreads, qproj_smem_bytes(), s, a, ak, av, n_heads) !=
               cudaSuccess) {
      return COBRA_ECUDA;
    }
  }
  if (stages & kScan) {
    const size_t smem =
        (size_t)kDecodeWarps * ((size_t)a.ring_bytes + decode_osm_bytes<G>() + decode_qfrag_bytes<G>() + kMaxStages * 8);
    static Granted granted;
    if (ensure_smem(decode_kernel<G>, smem, granted) != COBRA_OK) return COBRA_ECUDA;
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_kernel<G>, kDecodeWarps * 32, smem) != cudaSuccess)
      return COBRA_ECUDA;
    per_sm = std::max(per_sm, 1);
    const int want = (n_items + kDecodeWarps - 1) / kDecodeWarps;
    const int grid = std::max(1, std::min(want, per_sm * sm_count()));
    // the work counter is 0 here: the plan writes it so, and every scan's last CTA resets it
    if (launch_pdl(decode_kernel<G>, (unsigned)grid, kDecodeWarps * 32, smem, s, a) != cudaSuccess) return COBRA_ECUDA;
  }
  if (stages & kCombine) {
    // one CTA per (layer, kv head) and run of kCombineVP / G sequences
    constexpr int spp = kCombineVP / G > 0 ? kCombineVP / G : 1;
    const long long grid = (long long)n_heads * ((n_seqs + spp - 1) / spp);
    if (grid > 0x7fffffffLL) return COBRA_EINVAL;
    // its prologue (mu_V, the L2 prefetch of W_V) overlaps the scan's tail
    if (launch_pdl(combine_kernel<G, kCombineVP>, (unsigned)grid, kHeadThreads, combine_smem_bytes<kCombineVP>(), s,
                   a) != cudaSuccess)
      return COBRA_ECUDA;
  }
  return COBRA_OK;
}

// Checks shared by the decode entry points and the kernel arguments they build.
cobra_status decode_args(const void* params, const cobra_decode_desc* d, const cobra_decode_info* info, const void* q,
                         const uint8_t* cache, const int* seq_lens, const int* page_table, float* out, void* workspace,
                         size_t ws_bytes, int stages, DecodeArgs& a) {
  if (!d || !info || !params || !workspace) return COBRA_EINVAL;
  if ((stages & kQproj) && !q) return COBRA_EINVAL;
  if ((stages & kScan) && (!cache || !seq_lens)) return COBRA_EINVAL;
  if ((stages & kCombine) && (!out || !seq_lens)) return COBRA_EINVAL;
  if (d->n_layers < 1 || d->n_kv_heads < 1 || d->n_seqs < 1 || (d->group != 4 && d->group != 8)) return COBRA_EINVAL;
  if (page_table && d->pages_per_seq < 1) return COBRA_EINVAL;
  if (!aligned(params, 256) || !aligned(workspace, 256) || (cache && !aligned(cache, 256)) || (out && !aligned(out, 4)) ||
      (q && !aligned(q, 2)))
    return COBRA_EALIGN;
  if (info->max_row_bytes < 0 || info->max_row_bytes > 16 * 128 * 8 || (info->max_row_bytes % 16)) return COBRA_EINVAL;
  if (info->max_stage_bytes < 0 || info->max_stage_bytes > 2 * 16 * 128 * 8) return COBRA_EINVAL;
  if (ws_bytes < sizeof(WsHeader)) return COBRA_ESPACE;
  if (info->n_groups < 1 || info->n_items < 1) return COBRA_EINVAL;
  a = DecodeArgs{};
  a.block = static_cast<const unsigned char*>(params);
  a.cache = cache;
  a.seq_lens = seq_lens;
  a.page_table = page_table;
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.out = out;
  a.ws = static_cast<unsigned char*>(workspace);
  a.q_sl = d->q_stride_layer;
  a.q_ss = d->q_stride_seq;
  a.o_sl = d->o_stride_layer;
  a.o_ss = d->o_stride_seq;
  a.rows_per_seq = d->rows_per_seq;
  a.pages_per_seq = d->pages_per_seq;
  a.one = kOneH2;
  const int rowb = info->max_row_bytes > 0 ? info->max_row_bytes : 16;
  // 8 KB of row staging per warp, or two of the largest rows if those are bigger.  Rows of
  // 12 KB and more get four (at most 48 KB, which keeps a CTA within shared memory): with such
  // rows the copies, not the warps, bound the scan, and three stages of a typical row pair for
  // 4 warps per SM beat one stage for 8 (a 4 bpd rate sweep measured 0.50 against 0.43 of the
  // HBM peak; at 3 bpd, with 10 KB rows, the opposite held).
  size_t ring = std::max<size_t>(8192, 2 * align_up((size_t)rowb, 128));
  if (rowb >= 12288) ring = std::max(ring, std::min<size_t>(4 * align_up((size_t)rowb, 128), 48 * 1024));
  a.ring_bytes = (int)ring;
  const long long n_heads = (long long)d->n_layers * d->n_kv_heads;
  if (n_heads * d->n_seqs != info->n_groups) return COBRA_EINVAL;  // plan made for another descriptor
  return COBRA_OK;
}

cobra_status decode_common(const void* params, const cobra_decode_desc* d, const cobra_decode_info* info, const void* q,
                           const uint8_t* cache, const int* seq_lens, const int* page_table, float* out,
                           void* workspace, size_t ws_bytes, void* stream, int stages,
                           const CompressArgs& ak = CompressArgs{}, const CompressArgs& av = CompressArgs{}) {
  DecodeArgs a;
  const cobra_status st =
      decode_args(params, d, info, q, cache, seq_lens, page_table, out, workspace, ws_bytes, stages, a);
  if (st != COBRA_OK) return st;
  cudaStream_t s = (cudaStream_t)stream;
  const long long n_heads = (long long)d->n_layers * d->n_kv_heads;
  if (d->group == 4) return launch_decode<4>(a, (int)n_heads, d->n_seqs, info->n_items, stages, s, false, ak, av);
  return launch_decode<8>(a, (int)n_heads, d->n_seqs, info->n_items, stages, s, false, ak, av);
}

// K-side append arguments that match the decode descriptor's K heads
cobra_status k_append_args(const void* params, const cobra_decode_desc* d, const cobra_compress_desc* kdesc,
                           const void* k_new, const int* pos, uint8_t* cache, const int* page_table, CompressArgs& ak) {
  if (!d || !kdesc) return COBRA_EINVAL;
  cobra_status st = append_args(params, kdesc, k_new, pos, cache, page_table, ak);
  if (st != COBRA_OK) return st;
  if (kdesc->side != 0 || kdesc->head0 != d->k_head0 || kdesc->layer_stride != d->layer_stride ||
      kdesc->n_layers != d->n_layers || kdesc->n_kv_heads != d->n_kv_heads || kdesc->n_seqs != d->n_seqs)
    return COBRA_EINVAL;
  return COBRA_OK;
}
}  // namespace

extern "C" cobra_status cobra_decode_attn(const void* params, const cobra_decode_desc* d, const cobra_decode_info* info,
                                          const void* q, const uint8_t* cache, const int* seq_lens,
                                          const int* page_table, float* out, void* workspace, size_t ws_bytes,
                                          void* stream) {
  if (!q || !cache || !seq_lens || !out) return COBRA_EINVAL;
  return decode_common(params, d, info, q, cache, seq_lens, page_table, out, workspace, ws_bytes, stream,
                       kQproj | kScan | kCombine);
}

extern "C" cobra_status cobra_decode_qproj(const void* params, const cobra_decode_desc* d, const cobra_decode_info* info,
                                           const void* q, void* workspace, size_t ws_bytes, void* stream) {
  return decode_common(params, d, info, q, nullptr, nullptr, nullptr, nullptr, workspace, ws_bytes, stream, kQproj);
}

extern "C" cobra_status cobra_decode_qproj_append(const void* params, const cobra_decode_desc* d,
                                                  const cobra_decode_info* info, const void* q,
                                                  const cobra_compress_desc* kdesc, const void* k_new, const int* pos,
                                                  uint8_t* cache, const int* page_table, void* workspace,
                                                  size_t ws_bytes, void* stream) {
  CompressArgs ak;
  cobra_status st = k_append_args(params, d, kdesc, k_new, pos, cache, page_table, ak);
  if (st != COBRA_OK) return st;
  st = decode_common(params, d, info, q, nullptr, nullptr, nullptr, nullptr, workspace, ws_bytes, stream, kQproj, ak);
  return st != COBRA_OK ? st : launch_status();
}

extern "C" cobra_status cobra_decode_step(const void* params, const cobra_decode_desc* d, const cobra_decode_info* info,
                                          const cobra_compress_desc* kdesc, const cobra_compress_desc* vdesc,
                                          const void* k_new, const void* v_new, const int* pos, const void* q,
                                          uint8_t* cache, const int* seq_lens, const int* page_table, float* out,
                                          void* workspace, size_t ws_bytes, void* stream) {
  if (!d || !vdesc || !q || !seq_lens || !out) return COBRA_EINVAL;
  CompressArgs ak, av;
  cobra_status st = k_append_args(params, d, kdesc, k_new, pos, cache, page_table, ak);
  if (st != COBRA_OK) return st;
  st = append_args(params, vdesc, v_new, pos, cache, page_table, av);
  if (st != COBRA_OK) return st;
  if (vdesc->side != 1 || vdesc->head0 != d->v_head0 || vdesc->layer_stride != d->layer_stride ||
      vdesc->n_layers != d->n_layers || vdesc->n_kv_heads != d->n_kv_heads || vdesc->n_seqs != d->n_seqs)
    return COBRA_EINVAL;
  // the V append runs in the query projection's launch (its second half of CTAs)
  return decode_common(params, d, info, q, cache, seq_lens, page_table, out, workspace, ws_bytes, stream,
                       kQproj | kScan | kCombine, ak, av);
}

extern "C" cobra_status cobra_decode_scan(const void* params, const cobra_decode_desc* d, const cobra_decode_info* info,
                                          const uint8_t* cache, const int* seq_lens, const int* page_table,
                                          void* workspace, size_t ws_bytes, void* stream) {
  return decode_common(params, d, info, nullptr, cache, seq_lens, page_table, nullptr, workspace, ws_bytes, stream,
                       kScan);
}

extern "C" cobra_status cobra_decode_combine(const void* params, const cobra_decode_desc* d,
                                             const cobra_decode_info* info, const int* seq_lens, float* out,
                                             void* workspace, size_t ws_bytes, void* stream) {
  return decode_common(params, d, info, nullptr, nullptr, seq_lens, nullptr, out, workspace, ws_bytes, stream,
                       kCombine);
}

// ---------------------------------------------------------------------------------------
// Decode attention with the rotary position embedding applied after reconstruction.
// ---------------------------------------------------------------------------------------
namespace {

constexpr int kRopeMaxPos = 1 << 22;

int smem_optin() {
  int dev = 0, n = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&n, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  return n;
}

template <int G>
cobra_status launch_rope(const DecodeArgs& a, const RopeArgs& ra0, int n_heads, int n_seqs, int n_groups,
                         int n_items, int max_row_bytes, int max_stage_bytes, cudaStream_t s) {
  RopeArgs ra = ra0;
  // a stage holds the channel tiles of a K row and a V row: the plan's largest, else a bound
  // from the largest row (at most 1792 bytes of tiles past a K row); the two stages of a warp
  // also hold its partial for the merge
  const size_t rowb = (size_t)std::max(max_row_bytes, 16);
  const size_t need = max_stage_bytes > 0 ? (size_t)max_stage_bytes
                                          : align_up(rowb + 1792, 128) + align_up(rowb, 128);
  const size_t stage = std::max<size_t>(align_up(need, 128), 2560);
  ra.stage_bytes = (int)stage;
  const size_t fixed = rope_fixed_bytes<G>(), per_warp = rope_warp_bytes<G>((int)stage);
  const long long room = (long long)smem_optin() - 1024 - (long long)fixed;
  const int nw = (int)std::min<long long>(kRopeMaxWarps, room > 0 ? room / (long long)per_warp : 0);
  if (nw < 1) return COBRA_EINVAL;  // code rows too large for the staging
  const size_t smem = fixed + (size_t)nw * per_warp;
  static Granted granted;
  if (ensure_smem(rope_scan_kernel<G>, smem, granted) != COBRA_OK) return COBRA_ECUDA;
  if (launch_pdl(rope_qprep_kernel<G>, (unsigned)n_heads, kHeadThreads, 0, s, a, ra) != cudaSuccess)
    return COBRA_ECUDA;
  // one CTA per SM over the groups; the work counter is 0 here (the plan writes it so, every
  // scan resets it)
  const int grid = std::max(1, std::min(n_groups, sm_count()));
  if (launch_pdl(rope_scan_kernel<G>, (unsigned)grid, nw * 32, smem, s, a, ra) != cudaSuccess) return COBRA_ECUDA;
  return launch_decode<G>(a, n_heads, n_seqs, n_items, kCombine, s);
}

}  // namespace

extern "C" cobra_status cobra_rope_table_bytes(int max_pos, size_t* bytes) {
  if (!bytes || max_pos < 1 || max_pos > kRopeMaxPos) return COBRA_EINVAL;
  *bytes = rope_table_floats((max_pos + kRopeFine - 1) / kRopeFine) * sizeof(float);
  return COBRA_OK;
}

extern "C" cobra_status cobra_rope_table(double theta, int max_pos, float* table, size_t table_bytes, void* stream) {
  size_t need = 0;
  cobra_status st = cobra_rope_table_bytes(max_pos, &need);
  if (st != COBRA_OK) return st;
  if (!table || !(theta > 0.0) || !(theta < 1e300)) return COBRA_EINVAL;
  if (!aligned(table, 16)) return COBRA_EALIGN;
  if (table_bytes < need) return COBRA_ESPACE;
  const int n_rows = kRopeFine + (max_pos + kRopeFine - 1) / kRopeFine;
  const int n = n_rows * (kD / 2);
  if (launch_pdl(rope_table_kernel, (unsigned)((n + 255) / 256), 256, 0, (cudaStream_t)stream, table, n_rows, theta) !=
      cudaSuccess)
    return COBRA_ECUDA;
  return launch_status();
}

extern "C" cobra_status cobra_decode_rope_attn(const void* params, const cobra_decode_desc* d,
                                               const cobra_decode_info* info, const void* q, const int* q_pos,
                                               const float* rope_table, int max_pos, const uint8_t* cache,
                                               const int* seq_lens, const int* page_table, float* out,
                                               void* workspace, size_t ws_bytes, void* stream) {
  if (!q || !cache || !seq_lens || !out || !rope_table) return COBRA_EINVAL;
  if (max_pos < 1 || max_pos > kRopeMaxPos) return COBRA_EINVAL;
  if (!aligned(rope_table, 16) || (q_pos && !aligned(q_pos, 4))) return COBRA_EALIGN;
  DecodeArgs a;
  const cobra_status st = decode_args(params, d, info, q, cache, seq_lens, page_table, out, workspace, ws_bytes,
                                      kQproj | kScan | kCombine, a);
  if (st != COBRA_OK) return st;
  RopeArgs ra{};
  ra.table = rope_table;
  ra.q_pos = q_pos;
  ra.n_coarse = (max_pos + kRopeFine - 1) / kRopeFine;
  const int n_heads = d->n_layers * d->n_kv_heads;
  cudaStream_t s = (cudaStream_t)stream;
  cobra_status r = d->group == 4
                       ? launch_rope<4>(a, ra, n_heads, d->n_seqs, info->n_groups, info->n_items,
                                        info->max_row_bytes, info->max_stage_bytes, s)
                       : launch_rope<8>(a, ra, n_heads, d->n_seqs, info->n_groups, info->n_items,
                                        info->max_row_bytes, info->max_stage_bytes, s);
  return r != COBRA_OK ? r : launch_status();
}

// ---------------------------------------------------------------------------------------
// Decode attention with library-owned scratch (no device allocation by anyone).
//
// Some callers cannot allocate device memory: code that runs where cudaMalloc is not allowed
// or not wanted (inside an allocator's own callbacks, in a process whose memory pool is
// fixed at start-up, or in a plugin that may not touch the device heap).  For them this entry
// point keeps the decode workspace in one fixed array compiled into the library instead of
// a caller buffer.  The array is kStaticScratchBytes long, lives on every GPU that loads the
// library until the process exits, and is shared by every call on that GPU.
// ---------------------------------------------------------------------------------------
namespace {

constexpr size_t kStaticScratchBytes = COBRA_STATIC_SCRATCH_BYTES;
static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

// Address of g_static_scratch per device, with the context it was looked up in: a device
// reset (cudaDeviceReset) or another context made current on the device gives the array a new
// address, so the lookup is repeated whenever the current context differs from the recorded one.
struct ScratchAddr {
  std::atomic<unsigned char*> ptr{nullptr};
  std::atomic<void*> ctx{nullptr};
};
ScratchAddr g_scratch_addr[kMaxDevices];

using CtxGetCurrentFn = CUresult (*)(CUcontext*);
CtxGetCurrentFn ctx_get_current() {
  static CtxGetCurrentFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<CtxGetCurrentFn>(p);
  }
  return fn;
}

// The host-side address of g_static_scratch on the current device (looked up with that device
// and context current; cudaGetSymbolAddress allocates nothing).
cobra_status static_scratch(unsigned char** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return COBRA_ECUDA;
  CtxGetCurrentFn get = ctx_get_current();
  CUcontext ctx = nullptr;
  ScratchAddr& slot = g_scratch_addr[dev];
  unsigned char* p = slot.ptr.load(std::memory_order_acquire);
  if (p && get && get(&ctx) == CUDA_SUCCESS && ctx == slot.ctx.load(std::memory_order_acquire)) {
    *out = p;
    return COBRA_OK;
  }
  void* addr = nullptr;
  if (cudaGetSymbolAddress(&addr, g_static_scratch) != cudaSuccess || !addr) return COBRA_ECUDA;
  ctx = nullptr;
  if (get) get(&ctx);
  slot.ctx.store(ctx, std::memory_order_release);
  slot.ptr.store(static_cast<unsigned char*>(addr), std::memory_order_release);
  *out = static_cast<unsigned char*>(addr);
  return COBRA_OK;
}

// Workspace layout for a one-chunk-per-group plan with room for any head (r_V <= 128).
struct StaticPlanSizes {
  size_t groups_off, items_off, hg_off, qt_off, part_off, total;
  int g_stride, part_stride;
};
StaticPlanSizes static_plan_sizes(int n_groups, int group) {
  StaticPlanSizes z{};
  z.g_stride = 4 + kD;
  z.part_stride = z.g_stride * group;
  size_t off = align_up(sizeof(WsHeader), 256);
  z.groups_off = off;
  off = align_up(off + sizeof(WsGroup) * (size_t)n_groups, 256);
  z.items_off = off;
  off = align_up(off + sizeof(WsItem) * (size_t)n_groups, 256);
  z.hg_off = off;
  off = align_up(off + sizeof(int) * (size_t)n_groups, 256);
  z.qt_off = off;
  off = align_up(off + (size_t)kQtStride * n_groups, 256);
  z.part_off = off;
  off = align_up(off + sizeof(float) * (size_t)z.part_stride * n_groups, 256);
  z.total = off;
  return z;
}

// Writes the plan (header, groups, items) into the scratch: every (seq, layer, kv head) is one
// chunk covering the sequence's whole capacity; the scan clips it to seq_lens.  Every field the
// kernels read is rewritten on each call, so nothing has to start at zero.
__global__ void static_plan_kernel(unsigned char* ws, const unsigned char* block, cobra_decode_desc d,
                                   StaticPlanSizes z, int n_groups, int cap_rows) {
  WsGroup* groups = reinterpret_cast<WsGroup*>(ws + z.groups_off);
  WsItem* items = reinterpret_cast<WsItem*>(ws + z.items_off);
  int* hg = reinterpret_cast<int*>(ws + z.hg_off);
  const int n_heads = reinterpret_cast<const BlockHeader*>(block)->n_heads;
  for (int g = blockIdx.x * blockDim.x + threadIdx.x; g < n_groups; g += gridDim.x * blockDim.x) {
    const int h = g % d.n_kv_heads, l = (g / d.n_kv_heads) % d.n_layers, s = g / (d.n_kv_heads * d.n_layers);
    int hk = d.k_head0 + l * d.layer_stride + h, hv = d.v_head0 + l * d.layer_stride + h;
    int rows = cap_rows;
    if (hk >= n_heads || hv >= n_heads) {
      // the descriptor names a head the parameter block does not have: report it (cobra_check
      // returns COBRA_EINVAL) and plan an empty chunk on head 0, so nothing reads past the
      // head table or the cache
      atomicOr(&g_status, 2u);
      hk = hv = 0;
      rows = 0;
    }
    groups[g] = WsGroup{s, l, h, g, 1, hk, hv, 0};
    items[g] = WsItem{g, 0, rows, g};
    hg[((size_t)l * d.n_kv_heads + h) * d.n_seqs + s] = g;
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    WsHeader hd;
    memset(&hd, 0, sizeof(hd));
    hd.magic = kWsMagic;
    hd.version = COBRA_VERSION;
    hd.n_groups = n_groups;
    hd.n_items = n_groups;
    hd.group = d.group;
    hd.n_layers = d.n_layers;
    hd.n_kv = d.n_kv_heads;
    hd.n_seqs = d.n_seqs;
    hd.groups_off = z.groups_off;
    hd.items_off = z.items_off;
    hd.hg_off = z.hg_off;
    hd.qt_off = z.qt_off;
    hd.part_off = z.part_off;
    hd.part_stride = z.part_stride;
    hd.g_stride = z.g_stride;
    hd.qt_stride = kQtStride;
    hd.max_rv = kD;
    hd.max_row_bytes = 16 * kD * 8;
    *reinterpret_cast<WsHeader*>(ws) = hd;
  }
}

}  // namespace

extern "C" cobra_status cobra_decode_attn_static(const void* params, const cobra_decode_desc* d, const void* q,
                                                 const uint8_t* cache, const int* seq_lens, const int* page_table,
                                                 float* out, void* stream) {
  if (!d || !params || !q || !cache || !seq_lens || !out) return COBRA_EINVAL;
  if (d->n_layers < 1 || d->n_kv_heads < 1 || d->n_seqs < 1 || (d->group != 4 && d->group != 8) ||
      d->layer_stride < d->n_kv_heads || d->k_head0 < 0 || d->v_head0 < 0)
    return COBRA_EINVAL;
  if (page_table ? d->pages_per_seq < 1 : d->rows_per_seq < 1) return COBRA_EINVAL;
  if (!aligned(params, 256) || !aligned(cache, 256) || !aligned(out, 4) || !aligned(q, 2)) return COBRA_EALIGN;
  const long long n_groups = (long long)d->n_seqs * d->n_layers * d->n_kv_heads;
  if (n_groups > (1LL << 24)) return COBRA_ESPACE;
  const StaticPlanSizes z = static_plan_sizes((int)n_groups, d->group);
  if (z.total > kStaticScratchBytes) return COBRA_ESPACE;  // does not fit the fixed scratch
  const int cap_rows = page_table ? 2 * d->pages_per_seq : d->rows_per_seq;
  if (cap_rows > 65535) return COBRA_EINVAL;
  unsigned char* ws = nullptr;
  cobra_status st = static_scratch(&ws);
  if (st != COBRA_OK) return st;
  cudaStream_t s = (cudaStream_t)stream;
  static_plan_kernel<<<(unsigned)std::min<long long>((n_groups + 255) / 256, 1024), 256, 0, s>>>(
      ws, static_cast<const unsigned char*>(params), *d, z, (int)n_groups, cap_rows);
  if (cudaGetLastError() != cudaSuccess) return COBRA_ECUDA;
  DecodeArgs a{};
  a.block = static_cast<const unsigned char*>(params);
  a.cache = cache;
  a.seq_lens = seq_lens;
  a.page_table = page_table;
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.out = out;
  a.ws = ws;
  a.q_sl = d->q_stride_layer;
  a.q_ss = d->q_stride_seq;
  a.o_sl = d->o_stride_layer;
  a.o_ss = d->o_stride_seq;
  a.rows_per_seq = d->rows_per_seq;
  a.pages_per_seq = d->pages_per_seq;
  a.one = kOneH2;
  a.ring_bytes = 2 * 16 * kD * 8;  // two rows of the largest head (r = 128, b = 8)
  const int n_heads = d->n_layers * d->n_kv_heads;
  if (d->group == 4) return launch_decode<4>(a, n_heads, d->n_seqs, (int)n_groups, kQproj | kScan | kCombine, s, true);
  return launch_decode<8>(a, n_heads, d->n_seqs, (int)n_groups, kQproj | kScan | kCombine, s, true);
}

namespace {
// One warp waits on a barrier that expects one arrival nobody makes.
__global__ void selftest_wait_kernel(uint64_t limit_ns) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(smem_addr(&bar), 1);
    fence_mbar_init();
  }
  __syncwarp();
  const bool ok = __all_sync(0xffffffffu, mbar_wait_bounded(smem_addr(&bar), 0, limit_ns));
  if (!ok && threadIdx.x == 0) atomicOr(&g_status, 1u);
}
}  // namespace

extern "C" cobra_status cobra_selftest_wait_timeout(unsigned long long limit_ns, void* stream) {
  if (limit_ns == 0 || limit_ns > 100000000ull) return COBRA_EINVAL;
  selftest_wait_kernel<<<1, 32, 0, (cudaStream_t)stream>>>((uint64_t)limit_ns);
  return launch_status();
}

extern "C" cobra_status cobra_check(void* stream) {
  if (cudaStreamSynchronize((cudaStream_t)stream) != cudaSuccess) return COBRA_ECUDA;
  unsigned int v = 0;
  if (cudaMemcpyFromSymbol(&v, g_status, sizeof(v)) != cudaSuccess) return COBRA_ECUDA;
  if (v) {
    const unsigned int zero = 0;
    if (cudaMemcpyToSymbol(g_status, &zero, sizeof(zero)) != cudaSuccess) return COBRA_ECUDA;
    return (v & 1u) ? COBRA_ETIMEOUT : COBRA_EINVAL;
  }
  return COBRA_OK;
}

extern "C" cobra_status cobra_measure_distortion(int n_heads, int n_tok, const float* x, const float* U,
                                                 const double* lam, const double* w, const float* mu,
                                                 const int8_t* signs, int n_r, const int* r_list, int n_b,
                                                 const int* b_list, float* coords, double* D, void* stream) {
  if (n_heads < 1 || n_heads > 65535 || n_tok < 1 || !x || !U || !lam || !w || !mu || !signs || !r_list ||
      !b_list || !coords || !D || n_r < 1 || n_r > kMeasureMaxR || n_b < 1 || n_b > kMeasureMaxB)
    return COBRA_EINVAL;
  if (!aligned(x, 4) || !aligned(U, 4) || !aligned(lam, 8) || !aligned(w, 8) || !aligned(mu, 4) ||
      !aligned(coords, 4) || !aligned(D, 8))
    return COBRA_EALIGN;
  MeasureArgs a{};
  a.x = x;
  a.U = U;
  a.lam = lam;
  a.w = w;
  a.mu = mu;
  a.signs = signs;
  a.coords = coords;
  a.D = D;
  a.n_tok = n_tok;
  a.n_r = n_r;
  a.n_b = n_b;
  for (int i = 0; i < n_r; ++i) {
    if (r_list[i] < 0 || r_list[i] > kD || (i > 0 && r_list[i] <= r_list[i - 1])) return COBRA_EINVAL;
    a.r[i] = r_list[i];
  }
  for (int j = 0; j < n_b; ++j) {
    if (b_list[j] < 1 || b_list[j] > 8) return COBRA_EINVAL;
    a.b[j] = b_list[j];
    if (cobra_loading_factor(b_list[j], &a.L[j]) != COBRA_OK) return COBRA_EINVAL;
  }
  cudaStream_t s = (cudaStream_t)stream;
  coords_kernel<<<dim3((unsigned)((n_tok + kCoordTok - 1) / kCoordTok), (unsigned)n_heads), 256, 0, s>>>(a);
  if (cudaGetLastError() != cudaSuccess) return COBRA_ECUDA;
  measure_kernel<<<dim3((unsigned)n_r, (unsigned)n_heads), 256, 0, s>>>(a);
  return launch_status();
}

extern "C" cobra_status cobra_calibrate_heads(int n_heads, int n_tok, const float* x, int n_q, const float* q,
                                              double* mu, double* lam, double* U, double* w, void* stream) {
  if (n_heads < 1 || n_heads > 0x7fffffff || n_tok < 1 || !x || !mu || !lam || !U || !w || n_q < 0 ||
      (n_q > 0 && !q))
    return COBRA_EINVAL;
  if (!aligned(x, 4) || (q && !aligned(q, 4)) || !aligned(mu, 8) || !aligned(lam, 8) || !aligned(U, 8) ||
      !aligned(w, 8))
    return COBRA_EALIGN;
  static Granted granted;
  if (ensure_smem(calib_kernel, calib_smem_bytes(), granted) != COBRA_OK) return COBRA_ECUDA;
  CalibArgs a{};
  a.x = x;
  a.q = n_q > 0 ? q : nullptr;
  a.mu = mu;
  a.lam = lam;
  a.U = U;
  a.w = w;
  a.n_tok = n_tok;
  a.n_q = n_q;
  calib_kernel<<<(unsigned)n_heads, kCalThreads, calib_smem_bytes(), (cudaStream_t)stream>>>(a);
  return launch_status();
}

