// accept.cu -- the greedy P-MTP acceptance kernel.
#include <climits>

#include "common.cuh"

namespace hpd {
namespace {

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

cudaError_t launch_accept(const __nv_bfloat16 *logits, const int32_t *drafts, int B, int m, int V,
                          int32_t *out_tokens, int32_t *accepted_len, cudaStream_t s) {
  accept_kernel<<<B, kAcceptThreads, 0, s>>>(logits, drafts, m, V, out_tokens, accepted_len);
  return cudaGetLastError();
}

}  // namespace hpd
