// merge_accept.cu -- the log-sum-exp merge of the split partials and the
// greedy P-MTP acceptance kernel.
#include <climits>

#include "common.cuh"

namespace hpd {
namespace {

// One warp per (query token, query head): combine the S_total partials
//   O = sum_s e^{lse_s - M} O_s / sum_s e^{lse_s - M},
//   lse = M + ln sum_s e^{lse_s - M},   M = max_s lse_s,
// skipping partials whose chunk had no visible key (lse_s = -inf).  The union
// of the chunks is exactly the branch's visible key set (Sec. 3.3), so the
// result equals one softmax over all of it.
template <int D>
__global__ void __launch_bounds__(256) merge_kernel(const MergeParams p) {
  constexpr int E = D / 32;  // values per lane
  const int lane = threadIdx.x & 31;
  const long long pair = (static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const long long n_pairs = static_cast<long long>(p.rows_total) * p.H_q;
  if (pair >= n_pairs) return;
  const float NEG_INF = -__int_as_float(0x7f800000);

  const float ls = lane < p.S_total ? p.l_part[lane * n_pairs + pair] : NEG_INF;
  float M = ls;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));

  float acc[E];
#pragma unroll
  for (int e = 0; e < E; ++e) acc[e] = 0.f;
  float lse_out = NEG_INF;
  if (M != NEG_INF) {
    const float w_lane = ls == NEG_INF ? 0.f : exp2f((ls - M) * kLog2e);
    float wsum = w_lane;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) wsum += __shfl_xor_sync(0xffffffffu, wsum, o);
    for (int s = 0; s < p.S_total; ++s) {
      const float w = __shfl_sync(0xffffffffu, w_lane, s);
      if (w == 0.f) continue;
      const float *src = p.o_part + (s * n_pairs + pair) * D + lane * E;
      if constexpr (E == 4) {
        const float4 v = *reinterpret_cast<const float4 *>(src);
        acc[0] += w * v.x; acc[1] += w * v.y; acc[2] += w * v.z; acc[3] += w * v.w;
      } else {
        const float2 v = *reinterpret_cast<const float2 *>(src);
        acc[0] += w * v.x; acc[1] += w * v.y;
      }
    }
    const float inv = 1.f / wsum;
#pragma unroll
    for (int e = 0; e < E; ++e) acc[e] *= inv;
    lse_out = M + logf(wsum);
  }
  __nv_bfloat16 *dst = p.out + pair * D + lane * E;
  if constexpr (E == 4) {
    uint2 w;
    w.x = pack_bf16x2(acc[0], acc[1]);
    w.y = pack_bf16x2(acc[2], acc[3]);
    *reinterpret_cast<uint2 *>(dst) = w;
  } else {
    *reinterpret_cast<uint32_t *>(dst) = pack_bf16x2(acc[0], acc[1]);
  }
  if (p.lse && lane == 0) p.lse[pair] = lse_out;
}

// ------------------------------------------------------------ acceptance --
constexpr int kAcceptThreads = 512;
constexpr int kAcceptUnroll = 8;

struct ArgBest {
  float v;
  int i;
};

// Keep the larger value; among equal values the lower index.  NaN never
// compares true, so it is never taken.
__device__ __forceinline__ void consider(ArgBest &b, float x, int i) {
  if (x > b.v || (x == b.v && i < b.i)) {
    b.v = x;
    b.i = i;
  }
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// One CTA per branch: the argmax of each of its m logits rows (16-byte
// streaming loads, kAcceptUnroll in flight per thread), then the prefix
// match of the drafts (Sec. 3.4; Algorithm 1, verification).
__global__ void __launch_bounds__(kAcceptThreads)
    accept_kernel(const __nv_bfloat16 *__restrict__ logits, const int32_t *__restrict__ drafts,
                  int m, int V, int32_t *__restrict__ out_tokens,
                  int32_t *__restrict__ accepted_len) {
  __shared__ float s_v[kAcceptThreads / 32];
  __shared__ int s_i[kAcceptThreads / 32];
  __shared__ int s_tok[64];
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const float NEG_INF = -__int_as_float(0x7f800000);

  for (int j = 0; j < m; ++j) {
    const __nv_bfloat16 *row = logits + (static_cast<size_t>(b) * m + j) * V;
    ArgBest best{NEG_INF, INT_MAX};
    const uintptr_t addr = reinterpret_cast<uintptr_t>(row);
    const int head = min(V, static_cast<int>(((16u - (addr & 15u)) & 15u) >> 1));
    const int nvec = (V - head) >> 3;
    const int tail = head + (nvec << 3);
    for (int i = tid; i < head; i += kAcceptThreads) consider(best, __bfloat162float(row[i]), i);
    const uint4 *vrow = reinterpret_cast<const uint4 *>(row + head);
    for (int v0 = tid; v0 < nvec; v0 += kAcceptThreads * kAcceptUnroll) {
      uint4 x[kAcceptUnroll];
#pragma unroll
      for (int u = 0; u < kAcceptUnroll; ++u) {
        const int v = v0 + u * kAcceptThreads;
        if (v < nvec) x[u] = __ldcs(vrow + v);
      }
#pragma unroll
      for (int u = 0; u < kAcceptUnroll; ++u) {
        const int v = v0 + u * kAcceptThreads;
        if (v < nvec) {
          const int i0 = head + (v << 3);
          consider(best, bf16_lo(x[u].x), i0 + 0);
          consider(best, bf16_hi(x[u].x), i0 + 1);
          consider(best, bf16_lo(x[u].y), i0 + 2);
          consider(best, bf16_hi(x[u].y), i0 + 3);
          consider(best, bf16_lo(x[u].z), i0 + 4);
          consider(best, bf16_hi(x[u].z), i0 + 5);
          consider(best, bf16_lo(x[u].w), i0 + 6);
          consider(best, bf16_hi(x[u].w), i0 + 7);
        }
      }
    }
    for (int i = tail + tid; i < V; i += kAcceptThreads) consider(best, __bfloat162float(row[i]), i);

#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, best.v, o);
      const int oi = __shfl_xor_sync(0xffffffffu, best.i, o);
      consider(best, ov, oi);
    }
    if (lane == 0) {
      s_v[warp] = best.v;
      s_i[warp] = best.i;
    }
    __syncthreads();
    if (warp == 0) {
      best.v = lane < kAcceptThreads / 32 ? s_v[lane] : NEG_INF;
      best.i = lane < kAcceptThreads / 32 ? s_i[lane] : INT_MAX;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, best.v, o);
        const int oi = __shfl_xor_sync(0xffffffffu, best.i, o);
        consider(best, ov, oi);
      }
      if (lane == 0) {
        const int tok = best.i == INT_MAX ? 0 : best.i;
        out_tokens[static_cast<size_t>(b) * m + j] = tok;
        s_tok[j] = tok;
      }
    }
    __syncthreads();
  }
  if (tid == 0) {
    int k = 0;
    while (k < m && drafts[static_cast<size_t>(b) * m + k] == s_tok[k]) ++k;
    accepted_len[b] = k;
  }
}

}  // namespace

cudaError_t launch_merge(const MergeParams &p, cudaStream_t s) {
  const long long n_pairs = static_cast<long long>(p.rows_total) * p.H_q;
  const long long blocks = (n_pairs * 32 + 255) / 256;
  if (blocks <= 0) return cudaSuccess;
  if (p.D == 64)
    merge_kernel<64><<<static_cast<unsigned>(blocks), 256, 0, s>>>(p);
  else
    merge_kernel<128><<<static_cast<unsigned>(blocks), 256, 0, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_accept(const __nv_bfloat16 *logits, const int32_t *drafts, int B, int m, int V,
                          int32_t *out_tokens, int32_t *accepted_len, cudaStream_t s) {
  accept_kernel<<<B, kAcceptThreads, 0, s>>>(logits, drafts, m, V, out_tokens, accepted_len);
  return cudaGetLastError();
}

}  // namespace hpd
