// tc_common.cuh -- pieces shared by the tcgen05 shared-prefix kernels:
// locating a CTA's row tile, the key range of a prefix split, one 128-key
// block of a row's online softmax, and TMA tensor-map encoding on the host.
#pragma once

#include <cudaTypedefs.h>

#include <mutex>

#include "common.cuh"
#include "sm100.cuh"

namespace hpd {
namespace tc {

constexpr int kRows = 128;  // stacked query rows of one tile (MMA M)
constexpr int kBlk = 128;   // keys per block (MMA N of S = Q K^T)
constexpr float kRescaleLog2 = 8.0f;  // tolerate a stale row max up to 2^8

// Warp 0 finds the page owning row-tile `tile` of KV head blockIdx.y, where
// page d has ceil(#branches(d) * m / tile_tokens) tiles, and writes
// {d, tile index within d, first branch, end branch} to info (-1: no tile).
__device__ __forceinline__ void locate_tile(const AttnParams &p, int tile, int tile_tokens,
                                            int *info) {
  const int lane = threadIdx.x & 31;
  int base = 0;
  for (int d0 = 0; d0 < p.n_docs; d0 += 32) {
    const int d = d0 + lane;
    int tiles = 0, b0 = 0, b1 = 0;
    if (d < p.n_docs) {
      b0 = min(max(p.branch_cu[d], 0), p.B);
      b1 = min(max(p.branch_cu[d + 1], 0), p.B);
      if (b1 < b0) {
        flag_error(p.err, HPD_DEVERR_BRANCH_CU);
        b1 = b0;
      }
      tiles = ceil_div_i((b1 - b0) * p.m, tile_tokens);
    }
    int incl = tiles;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    const int excl = incl - tiles;
    if (tiles > 0 && tile >= base + excl && tile < base + incl) {
      info[0] = d;
      info[1] = tile - base - excl;
      info[2] = b0;
      info[3] = b1;
    }
    base += __shfl_sync(0xffffffffu, incl, 31);
    if (base > tile) break;
  }
}

// Key range of prefix split `split` of a page with P_d keys: the page's
// ceil(P_d / 128) blocks are dealt out as evenly as possible.
__device__ __forceinline__ void split_range(int P_d, int S_p, int split, int &k_begin,
                                            int &k_end) {
  const int nb = ceil_div_i(P_d, kBlk);
  const int b0 = static_cast<int>(static_cast<long long>(split) * nb / S_p);
  const int b1 = static_cast<int>(static_cast<long long>(split + 1) * nb / S_p);
  k_begin = b0 * kBlk;
  k_end = min(P_d, b1 * kBlk);
}

// One 128-key block of a row's online softmax (base 2, scaled scores).
// v holds the raw scores of keys key0 .. key0+127; keys >= lim are masked.
// Writes the bf16 probabilities relative to the (possibly stale) running
// max into pk, updates m_run / l_run, and returns the factor by which the
// row's accumulated output must be rescaled (1 if unchanged).
__device__ __forceinline__ float softmax_block(uint32_t (&v)[kBlk], int key0, int lim, float sl2,
                                               float &m_run, float &l_run,
                                               uint32_t (&pk)[kBlk / 2]) {
  const float NEG_INF = -__int_as_float(0x7f800000);
  float mx8[8];
#pragma unroll
  for (int a = 0; a < 8; ++a) mx8[a] = NEG_INF;
  const bool fast = sl2 > 0.f && key0 + kBlk <= lim;  // whole block visible
  if (fast) {
    // max of the raw scores, scaled afterwards (a positive scale keeps order)
#pragma unroll
    for (int c = 0; c < kBlk; ++c) mx8[c & 7] = fmaxf(mx8[c & 7], __uint_as_float(v[c]));
  } else {
#pragma unroll
    for (int c = 0; c < kBlk; ++c) {
      const float f = key0 + c < lim ? __uint_as_float(v[c]) * sl2 : NEG_INF;
      v[c] = __float_as_uint(f);
      mx8[c & 7] = fmaxf(mx8[c & 7], f);
    }
  }
  float mx = fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                   fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7])));
  if (fast) mx *= sl2;
  const float m_new = mx > m_run + kRescaleLog2 ? mx : m_run;
  const float base = m_new == NEG_INF ? 0.f : m_new;
  const float alpha = m_new == m_run ? 1.f : fast_exp2(m_run - base);
  float sum8[8];
#pragma unroll
  for (int a = 0; a < 8; ++a) sum8[a] = 0.f;
  if (fast) {
#pragma unroll
    for (int c = 0; c < kBlk; c += 2) {
      const float e0 = fast_exp2(fmaf(__uint_as_float(v[c]), sl2, -base));
      const float e1 = fast_exp2(fmaf(__uint_as_float(v[c + 1]), sl2, -base));
      sum8[(c >> 1) & 7] += e0 + e1;
      pk[c / 2] = pack_bf16x2(e0, e1);
    }
  } else {
#pragma unroll
    for (int c = 0; c < kBlk; c += 2) {
      const float e0 = fast_exp2(__uint_as_float(v[c]) - base);
      const float e1 = fast_exp2(__uint_as_float(v[c + 1]) - base);
      sum8[(c >> 1) & 7] += e0 + e1;
      pk[c / 2] = pack_bf16x2(e0, e1);
    }
  }
  const float sum = ((sum8[0] + sum8[1]) + (sum8[2] + sum8[3])) +
                    ((sum8[4] + sum8[5]) + (sum8[6] + sum8[7]));
  l_run = l_run * alpha + sum;
  m_run = m_new;
  return alpha;
}

// ------------------------------------------------------------------ host --
inline PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// 3-D bf16 tensor map over [d2][d1][d0] (d0 contiguous) with a
// (b0, b1, b2) box and 128-byte swizzle.
inline cudaError_t make_map(CUtensorMap *map, const void *base, uint64_t d0, uint64_t d1,
                            uint64_t d2, uint32_t b0, uint32_t b1, uint32_t b2) {
  auto fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  const cuuint64_t dims[3] = {d0, d1, d2};
  const cuuint64_t strides[2] = {d0 * 2, d0 * d1 * 2};
  const cuuint32_t box[3] = {b0, b1, b2};
  const cuuint32_t es[3] = {1, 1, 1};
  const CUresult r =
      fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box,
         es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
         CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// Maps of Q (box: 64 columns x G heads x 128/G tokens = one 128-row tile)
// and of the prefix K / V (box: 64 columns x 1 head x 128 keys).
inline cudaError_t make_prefix_maps(const AttnParams &p, CUtensorMap *tq, CUtensorMap *tk,
                                    CUtensorMap *tv) {
  const int D = p.D, G = p.G;
  cudaError_t e = make_map(tq, p.q, D, p.H_q, static_cast<uint64_t>(p.rows_total), 64, G,
                           kRows / G);
  if (e != cudaSuccess) return e;
  const bool has_prefix = p.prefix_tokens > 0;
  const uint64_t T = has_prefix ? static_cast<uint64_t>(p.prefix_tokens) : 1;
  e = make_map(tk, has_prefix ? p.prefix_k : p.k_cache, D, p.H_kv, T, 64, 1, kBlk);
  if (e != cudaSuccess) return e;
  return make_map(tv, has_prefix ? p.prefix_v : p.v_cache, D, p.H_kv, T, 64, 1, kBlk);
}

}  // namespace tc
}  // namespace hpd
