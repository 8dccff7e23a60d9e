// tc_common.cuh -- pieces of the tcgen05 branch-attention kernel: half of a
// 128-key block of a row's online softmax, and TMA tensor-map encoding on
// the host.
#pragma once

#include <cudaTypedefs.h>

#include <mutex>

#include "common.cuh"
#include "sm100.cuh"

namespace hpd {
namespace tc {

// max(a, b, c) in one instruction (three-input max.f32, sm_100 and later).
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

constexpr int kRows = 128;  // stacked query rows of one tile (MMA M)
constexpr int kBlk = 128;   // keys per block (MMA N of S = Q K^T)
constexpr float kRescaleLog2 = 8.0f;  // tolerate a stale row max up to 2^8

// Half of one 128-key block of a row's online softmax: this thread owns the
// 64 columns [64 h, 64 h + 64) of its row; the thread of the other half (the
// same TMEM lane, another warpgroup) owns the rest.  s_addr is this thread's
// lane at the block's first column; lo / hi bound the row's visible columns
// in block coordinates.  xchg(max of my visible scaled scores) returns the
// row max over both halves; it must synchronise the two halves, which also
// orders every P store of either half after both have read their scores
// (P half h lands in packed columns [32 h, 32 h + 32), over scores of half 0).
// Both halves apply the same running max, so O's two column halves and the
// two partial sums l_half stay consistent.  Returns the rescale factor of O.
// Warp-collective (tcgen05.ld / st).
template <class Xchg>
__device__ __forceinline__ float softmax_half_tmem(uint32_t s_addr, int h, int lo, int hi,
                                                   float sl2, float &m_run, float &l_half,
                                                   Xchg xchg) {
  using namespace sm100;
  const float NEG_INF = -__int_as_float(0x7f800000);
  constexpr int kH = kBlk / 2;
  lo = max(lo - h * kH, 0);
  hi = min(hi - h * kH, kH);
  const bool all_empty = __all_sync(0xffffffffu, hi <= lo);
  const bool all_full = __all_sync(0xffffffffu, lo == 0 && hi == kH);
  uint32_t v[kH];
  float mx = NEG_INF;
  // A positive scale keeps the order of the scores, so the maximum can be
  // taken over the raw scores and an invisible score can simply become -inf
  // in place (its exponential is then 0): one select per score instead of a
  // visibility test in both loops below.
  const bool raw = sl2 > 0.f;
  if (!all_empty) {
    tmem_ld32(s_addr + h * kH, v);
    tmem_ld32(s_addr + h * kH + 32, v + 32);
    tmem_ld_wait();
    float mx8[8];
#pragma unroll
    for (int a = 0; a < 8; ++a) mx8[a] = NEG_INF;
    if (raw) {
      if (!all_full) {
        // bit c of vis: column c of this half is visible
        auto below = [](int n) -> uint64_t {
          return n <= 0 ? 0ull : n >= 64 ? ~0ull : (1ull << n) - 1ull;
        };
        const uint64_t vis = below(hi) & ~below(lo);
        const uint32_t vis0 = static_cast<uint32_t>(vis), vis1 = static_cast<uint32_t>(vis >> 32);
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          v[c] = (vis0 & (1u << c)) ? v[c] : 0xff800000u;
          v[c + 32] = (vis1 & (1u << c)) ? v[c + 32] : 0xff800000u;
        }
      }
#pragma unroll
      for (int c = 0; c < kH; c += 16)
#pragma unroll
        for (int a = 0; a < 8; ++a)
          mx8[a] = fmax3(mx8[a], __uint_as_float(v[c + 2 * a]), __uint_as_float(v[c + 2 * a + 1]));
    } else {
#pragma unroll
      for (int c = 0; c < kH; c += 16)
#pragma unroll
        for (int a = 0; a < 8; ++a) {
          const int c0 = c + 2 * a;
          const float x0 = c0 >= lo && c0 < hi ? __uint_as_float(v[c0]) * sl2 : NEG_INF;
          const float x1 = c0 + 1 >= lo && c0 + 1 < hi ? __uint_as_float(v[c0 + 1]) * sl2 : NEG_INF;
          mx8[a] = fmax3(mx8[a], x0, x1);
        }
    }
    mx = fmax3(fmax3(mx8[0], mx8[1], mx8[2]), fmax3(mx8[3], mx8[4], mx8[5]),
               fmaxf(mx8[6], mx8[7]));
    if (raw) mx *= sl2;
  }
  mx = xchg(mx);
  const float m_new = mx > m_run + kRescaleLog2 ? mx : m_run;
  const float base = m_new == NEG_INF ? 0.f : m_new;
  const float alpha = m_new == m_run ? 1.f : fast_exp2(m_run - base);
  float sum = 0.f;
  uint32_t pk[16];
  if (all_empty) {
#pragma unroll
    for (int c = 0; c < 16; ++c) pk[c] = 0u;
    tmem_st16(s_addr + h * 32, pk);
    tmem_st16(s_addr + h * 32 + 16, pk);
  } else {
    const float2 sl2x2 = make_float2(sl2, sl2), nbase2 = make_float2(-base, -base);
    float2 sum4[4];
#pragma unroll
    for (int a = 0; a < 4; ++a) sum4[a] = make_float2(0.f, 0.f);
    if (all_full || raw) {
#pragma unroll
      for (int ch = 0; ch < 2; ++ch) {
#pragma unroll
        for (int c = 0; c < 32; c += 2) {
          const int col = ch * 32 + c;
          const float2 x = make_float2(__uint_as_float(v[col]), __uint_as_float(v[col + 1]));
          const float2 arg = __ffma2_rn(x, sl2x2, nbase2);
          const float2 e = make_float2(fast_exp2(arg.x), fast_exp2(arg.y));
          sum4[(c >> 1) & 3] = __fadd2_rn(sum4[(c >> 1) & 3], e);
          pk[c / 2] = pack_bf16x2(e.x, e.y);
        }
        tmem_st16(s_addr + h * 32 + ch * 16, pk);
      }
    } else {
#pragma unroll
      for (int ch = 0; ch < 2; ++ch) {
#pragma unroll
        for (int c = 0; c < 32; c += 2) {
          const int col = ch * 32 + c;
          const float2 x = make_float2(__uint_as_float(v[col]), __uint_as_float(v[col + 1]));
          const float2 arg = __ffma2_rn(x, sl2x2, nbase2);
          float2 e;
          e.x = col >= lo && col < hi ? fast_exp2(arg.x) : 0.f;
          e.y = col + 1 >= lo && col + 1 < hi ? fast_exp2(arg.y) : 0.f;
          sum4[(c >> 1) & 3] = __fadd2_rn(sum4[(c >> 1) & 3], e);
          pk[c / 2] = pack_bf16x2(e.x, e.y);
        }
        tmem_st16(s_addr + h * 32 + ch * 16, pk);
      }
    }
    const float2 s01 = __fadd2_rn(sum4[0], sum4[1]), s23 = __fadd2_rn(sum4[2], sum4[3]);
    const float2 s03 = __fadd2_rn(s01, s23);
    sum = s03.x + s03.y;
  }
  l_half = l_half * alpha + sum;
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

// 4-D bf16 tensor map over the paged cache [pages][16][H_kv][D]: one box
// is box_pages consecutive pages of one KV head (64 columns x 1 head x 16
// tokens x box_pages pages), rows in page-then-slot order.
inline cudaError_t make_page_map(CUtensorMap *map, const void *base, int D, int H_kv,
                                 int num_pages, int box_pages = 1) {
  auto fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  const cuuint64_t dims[4] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(H_kv),
                              static_cast<cuuint64_t>(kPage), static_cast<cuuint64_t>(num_pages)};
  const cuuint64_t row = static_cast<cuuint64_t>(D) * 2;
  const cuuint64_t strides[3] = {row, row * H_kv, row * H_kv * kPage};
  const cuuint32_t box[4] = {64, 1, static_cast<cuuint32_t>(kPage),
                             static_cast<cuuint32_t>(box_pages)};
  const cuuint32_t es[4] = {1, 1, 1, 1};
  const CUresult r =
      fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims, strides, box,
         es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
         CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// Map of Q ([B m][H_q][D]): one box is 64 columns x G heads x 128 / G
// tokens, i.e. one 128-row tile of stacked query rows (row = token x G +
// head within the KV group) in the layout of a 128-key K block; rows past
// the last token read zeros.
inline cudaError_t make_q_map(const AttnParams &p, CUtensorMap *tq) {
  return make_map(tq, p.q, p.D, p.H_q, static_cast<uint64_t>(p.rows_total), 64, p.G, kRows / p.G);
}

// K and V maps of the contiguous prefix ([tokens][H_kv][D], one KV head x
// 128 keys x 64 columns per box); the paged cache stands in when there is
// no prefix at all (the maps are then never used).
inline cudaError_t make_prefix_maps(const AttnParams &p, CUtensorMap *tk, CUtensorMap *tv) {
  const int D = p.D;
  const bool has_prefix = p.prefix_tokens > 0 && !p.prefix_page_table;  // paged: page maps
  const uint64_t T = has_prefix ? static_cast<uint64_t>(p.prefix_tokens) : 1;
  cudaError_t e = make_map(tk, has_prefix ? p.prefix_k : p.k_cache, D, p.H_kv, T, 64, 1, kBlk);
  if (e != cudaSuccess) return e;
  return make_map(tv, has_prefix ? p.prefix_v : p.v_cache, D, p.H_kv, T, 64, 1, kBlk);
}

}  // namespace tc
}  // namespace hpd
