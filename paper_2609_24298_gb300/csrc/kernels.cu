// libcobra device entry points: argument checks and launches for compress, append and
// decode attention, plus the device status check.
#include <cuda_runtime.h>

#include <algorithm>

#include "../../include/cobra.h"
#include "common.cuh"
#include "compress.cuh"
#include "decode.cuh"

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
  static bool attr = false;
  if (!attr) {
    if (cudaFuncSetAttribute(compress_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kCompressSmem) != cudaSuccess)
      return COBRA_ECUDA;
    attr = true;
  }
  CompressArgs a{};
  a.block = static_cast<const unsigned char*>(params);
  a.x = static_cast<const __nv_bfloat16*>(x);
  a.cache = cache;
  a.page_table = page_table;
  a.sl = d->x_stride_layer;
  a.ss = d->x_stride_seq;
  a.st = d->x_stride_tok;
  a.sh = d->x_stride_head;
  a.head0 = d->head0;
  a.layer_stride = d->layer_stride;
  a.n_layers = d->n_layers;
  a.n_kv = d->n_kv_heads;
  a.side = d->side;
  a.n_seqs = d->n_seqs;
  a.rows_per_seq = d->rows_per_seq;
  a.pages_per_seq = d->pages_per_seq;
  a.t0 = t0;
  a.n_tok = n_tok;
  const int heads = d->n_layers * d->n_kv_heads;
  const long long tiles = (long long)d->n_seqs * ((n_tok + kRowTokens - 1) / kRowTokens);
  // about two waves of CTAs, each CTA converting its head's basis once
  long long chunks = std::max(1LL, (2LL * sm_count() + heads - 1) / heads);
  chunks = std::min(chunks, tiles);
  a.chunks = (int)chunks;
  const long long grid = (long long)heads * chunks;
  if (grid > 0x7fffffffLL) return COBRA_EINVAL;
  compress_kernel<<<(unsigned)grid, kCompressThreads, kCompressSmem, (cudaStream_t)stream>>>(a);
  return launch_status();
}

extern "C" cobra_status cobra_append(const void* params, const cobra_compress_desc* d, const void* x, const int* pos,
                                     uint8_t* cache, const int* page_table, void* stream) {
  cobra_status st = check_compress_desc(d);
  if (st != COBRA_OK) return st;
  if (!params || !x || !pos || !cache) return COBRA_EINVAL;
  if (!aligned(params, 256) || !aligned(cache, 256) || !aligned(x, 2)) return COBRA_EALIGN;
  if (page_table && d->pages_per_seq < 1) return COBRA_EINVAL;
  CompressArgs a{};
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
  const long long warps = (long long)d->n_layers * d->n_kv_heads * d->n_seqs;
  const long long grid = (warps + 3) / 4;
  if (grid > 0x7fffffffLL) return COBRA_EINVAL;
  append_kernel<<<(unsigned)grid, 128, 0, (cudaStream_t)stream>>>(a);
  return launch_status();
}

namespace {
enum Stage { kQproj = 1, kScan = 2, kCombine = 4 };

template <int G>
cobra_status launch_decode(const DecodeArgs& a, int n_groups, int n_items, int stages, cudaStream_t s) {
  if (stages & kQproj) {
    qproj_kernel<G><<<n_groups, 128, 0, s>>>(a);
    if (cudaGetLastError() != cudaSuccess) return COBRA_ECUDA;
  }
  if (stages & kScan) {
    const size_t smem = (size_t)kDecodeWarps * ((size_t)a.ring_bytes + (size_t)(G / 4) * 8 * 32 * 16 + kMaxStages * 8);
    static size_t attr_set = 0;
    if (smem > attr_set) {
      if (cudaFuncSetAttribute(decode_kernel<G>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
        return COBRA_ECUDA;
      attr_set = smem;
    }
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_kernel<G>, kDecodeWarps * 32, smem) != cudaSuccess)
      return COBRA_ECUDA;
    per_sm = std::max(per_sm, 1);
    const int want = (n_items + kDecodeWarps - 1) / kDecodeWarps;
    const int grid = std::max(1, std::min(want, per_sm * sm_count()));
    decode_kernel<G><<<grid, kDecodeWarps * 32, smem, s>>>(a);
    if (cudaGetLastError() != cudaSuccess) return COBRA_ECUDA;
  }
  if (stages & kCombine) {
    combine_kernel<G><<<n_groups, 128, 0, s>>>(a);
    if (cudaGetLastError() != cudaSuccess) return COBRA_ECUDA;
  }
  return COBRA_OK;
}

cobra_status decode_common(const void* params, const cobra_decode_desc* d, const cobra_decode_info* info, const void* q,
                           const uint8_t* cache, const int* seq_lens, const int* page_table, float* out,
                           void* workspace, size_t ws_bytes, void* stream, int stages) {
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
  if (ws_bytes < sizeof(WsHeader)) return COBRA_ESPACE;
  if (info->n_groups < 1 || info->n_items < 1) return COBRA_EINVAL;
  DecodeArgs a{};
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
  const int rowb = info->max_row_bytes > 0 ? info->max_row_bytes : 16;
  // 8 KB of row staging per warp, or two of the largest rows if those are bigger
  a.ring_bytes = (int)std::max<size_t>(8192, 2 * align_up((size_t)rowb, 128));
  cudaStream_t s = (cudaStream_t)stream;
  if (d->group == 4) return launch_decode<4>(a, info->n_groups, info->n_items, stages, s);
  return launch_decode<8>(a, info->n_groups, info->n_items, stages, s);
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
