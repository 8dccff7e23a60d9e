// merge.cu -- log-sum-exp merge of the key splits of the tcgen05 branch-
// attention kernel, used when a (page, KV head) row tile is split across
// several CTAs.
//
// Each split s holds, for every (query token, query head), the softmax over
// its share of the visible keys: O_s normalised and lse_s (natural log,
// -inf for no visible key).  The splits partition the branch's visible key
// set (Sec. 3.3), so
//   out = sum_s e^{lse_s - M} O_s / sum_s e^{lse_s - M},
//   lse = M + ln sum_s e^{lse_s - M},   M = max_s lse_s,
// equals one softmax over all of it; no visible key anywhere gives out = 0
// and lse = -inf.
#include "common.cuh"

namespace hpd {
namespace {

constexpr int kMaxSplits = 8;

// One warp per (token, head); lane s loads split s's lse, every lane loads
// D/32 columns of all splits with the loads in flight together.
template <int D>
__global__ void __launch_bounds__(256) merge_splits_kernel(const AttnParams p) {
  constexpr int E = D / 32;
  const int lane = threadIdx.x & 31;
  const long long n_pairs = static_cast<long long>(p.rows_total) * p.H_q;
  const long long pair = (static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  pdl_wait();  // the partial results of the attention kernel
  if (pair >= n_pairs) return;
  const float NEG_INF = -__int_as_float(0x7f800000);
  const int S = p.S_p;

  const float ls = lane < S ? p.l_part[lane * n_pairs + pair] : NEG_INF;
  float M = ls;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
  const float w_lane = (M == NEG_INF || ls == NEG_INF) ? 0.f : __expf(ls - M);
  float wsum = w_lane;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) wsum += __shfl_xor_sync(0xffffffffu, wsum, o);

  float v[kMaxSplits][E];
  float w[kMaxSplits];
#pragma unroll
  for (int s = 0; s < kMaxSplits; ++s) {
    w[s] = __shfl_sync(0xffffffffu, w_lane, s);
    const float *src = p.o_part + (s * n_pairs + pair) * D + lane * E;
    if (s < S && w[s] != 0.f) {
      if constexpr (E == 4) {
        const float4 x = *reinterpret_cast<const float4 *>(src);
        v[s][0] = x.x; v[s][1] = x.y; v[s][2] = x.z; v[s][3] = x.w;
      } else {
        const float2 x = *reinterpret_cast<const float2 *>(src);
        v[s][0] = x.x; v[s][1] = x.y;
      }
    } else {
#pragma unroll
      for (int e = 0; e < E; ++e) v[s][e] = 0.f;
    }
  }
  float acc[E];
#pragma unroll
  for (int e = 0; e < E; ++e) {
    acc[e] = 0.f;
#pragma unroll
    for (int s = 0; s < kMaxSplits; ++s) acc[e] += w[s] * v[s][e];
  }
  const float inv = wsum > 0.f ? 1.f / wsum : 0.f;
  __nv_bfloat16 *dst = p.out + pair * D + lane * E;
  if constexpr (E == 4) {
    uint2 x;
    x.x = pack_bf16x2(acc[0] * inv, acc[1] * inv);
    x.y = pack_bf16x2(acc[2] * inv, acc[3] * inv);
    *reinterpret_cast<uint2 *>(dst) = x;
  } else {
    *reinterpret_cast<uint32_t *>(dst) = pack_bf16x2(acc[0] * inv, acc[1] * inv);
  }
  if (p.lse && lane == 0) p.lse[pair] = M == NEG_INF ? NEG_INF : M + logf(wsum);
}

}  // namespace

cudaError_t launch_merge_splits(const AttnParams &p, bool overlap, cudaStream_t s) {
  if (p.S_p > kMaxSplits) return cudaErrorInvalidValue;
  const long long n_pairs = static_cast<long long>(p.rows_total) * p.H_q;
  const long long blocks = (n_pairs * 32 + 255) / 256;
  if (blocks <= 0) return cudaSuccess;
  const dim3 grid(static_cast<unsigned>(blocks));
  return p.D == 64 ? launch_kernel(overlap, merge_splits_kernel<64>, grid, dim3(256), 0, s, p)
                   : launch_kernel(overlap, merge_splits_kernel<128>, grid, dim3(256), 0, s, p);
}

}  // namespace hpd
