// accept.cu -- greedy verification of the P-MTP drafts (Sec. 3.4; the
// verification step of Algorithm 1):
//   t*_{b,j} = argmax_v logits[b][j][v]   (lowest index among equal maxima;
//                                           NaN never wins; all-NaN row -> 0)
//   n_acc_b  = largest k <= m with drafts[b][i] == t*_{b,i} for all i < k
//
// One thread-block cluster per branch, one CTA per logits row (rows beyond
// the cluster size are taken in turn).  Each CTA streams its row with
// 16-byte loads, reduces (value, index) over the CTA, and writes its token
// to the output and into the leader CTA's shared memory (distributed shared
// memory, written only after a cluster barrier shows that every CTA of the
// cluster runs); after a second cluster barrier the leader matches the
// drafts.
#include <cooperative_groups.h>

#include <climits>

#include "common.cuh"

namespace cg = cooperative_groups;

namespace hpd {
namespace {

constexpr int kAcceptThreads = 256;
constexpr int kAcceptUnroll = 8;
constexpr int kMaxCluster = 8;  // portable cluster size
constexpr int kMaxRows = 64;

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
// The same for a thread's own scan, whose indices only grow: a later equal
// value never wins, so the strict comparison suffices.
__device__ __forceinline__ void consider_next(ArgBest &b, float x, int i) {
  if (x > b.v) {
    b.v = x;
    b.i = i;
  }
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// Argmax of one row of V bf16 values, reduced over the CTA (valid in thread 0).
// s_none: a shared word, set when no value above -inf was found.
__device__ __forceinline__ int row_argmax(const __nv_bfloat16 *row, int V, float *s_v, int *s_i,
                                          int *s_none) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const float NEG_INF = -__int_as_float(0x7f800000);
  ArgBest best{NEG_INF, INT_MAX};
  const uintptr_t addr = reinterpret_cast<uintptr_t>(row);
  const int head = min(V, static_cast<int>(((16u - (addr & 15u)) & 15u) >> 1));
  const int nvec = (V - head) >> 3;
  const int tail = head + (nvec << 3);
  // each thread visits its indices in increasing order: head, vectors, tail
  for (int i = tid; i < head; i += kAcceptThreads) consider_next(best, __bfloat162float(row[i]), i);
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
        consider_next(best, bf16_lo(x[u].x), i0 + 0);
        consider_next(best, bf16_hi(x[u].x), i0 + 1);
        consider_next(best, bf16_lo(x[u].y), i0 + 2);
        consider_next(best, bf16_hi(x[u].y), i0 + 3);
        consider_next(best, bf16_lo(x[u].z), i0 + 4);
        consider_next(best, bf16_hi(x[u].z), i0 + 5);
        consider_next(best, bf16_lo(x[u].w), i0 + 6);
        consider_next(best, bf16_hi(x[u].w), i0 + 7);
      }
    }
  }
  for (int i = tail + tid; i < V; i += kAcceptThreads)
    consider_next(best, __bfloat162float(row[i]), i);
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
    if (lane == 0) *s_none = best.i == INT_MAX ? INT_MAX : -1;
  }
  __syncthreads();  // s_v / s_i are reused by the next row
  if (*s_none == INT_MAX) {
    // No value above -inf (the strict scan never takes a -inf): the maximum
    // is -inf if the row holds one, at its first position (rare path).
    __syncthreads();  // every thread has read the word before it is reused
    for (int i = tid; i < V; i += kAcceptThreads)
      if (__bfloat162float(row[i]) == NEG_INF) {
        atomicMin(s_none, i);
        break;
      }
    __syncthreads();
    best.i = *s_none;
    __syncthreads();  // read before the next row's flag
  }
  return best.i == INT_MAX ? 0 : best.i;
}

// Split cluster barrier (every thread of every CTA of the cluster arrives
// once, then waits for the phase).
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
  asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
}

// grid (cluster size * B), cluster (cluster size, 1, 1): cluster = branch.
__global__ void __launch_bounds__(kAcceptThreads)
    accept_cluster_kernel(const __nv_bfloat16 *__restrict__ logits,
                          const int32_t *__restrict__ drafts, int m, int V,
                          int32_t *__restrict__ out_tokens, int32_t *__restrict__ accepted_len) {
  __shared__ float s_v[kAcceptThreads / 32];
  __shared__ int s_i[kAcceptThreads / 32];
  __shared__ int s_tok[kMaxRows];  // used in the leader CTA
  __shared__ int s_none;
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = static_cast<int>(cluster.block_rank());
  const int cs = static_cast<int>(cluster.num_blocks());
  const int b = blockIdx.x / cs;
  int *leader_tok = cluster.map_shared_rank(s_tok, 0);
  // The leader's shared memory may be written only once the leader CTA is
  // known to run: a split cluster barrier, whose arrive comes first and whose
  // wait comes just before the first remote write, so that the first row's
  // scan overlaps the other CTAs' start.
  cluster_arrive_relaxed();
  bool joined = false;
  for (int j = rank; j < m; j += cs) {
    const int tok = row_argmax(logits + (static_cast<size_t>(b) * m + j) * V, V, s_v, s_i, &s_none);
    if (!joined) {  // uniform over the CTA
      cluster_wait();
      joined = true;
    }
    if (threadIdx.x == 0) {
      out_tokens[static_cast<size_t>(b) * m + j] = tok;
      leader_tok[j] = tok;
    }
  }
  if (!joined) cluster_wait();
  cluster.sync();  // every row's token is in the leader's shared memory
  if (rank == 0 && threadIdx.x == 0) {
    int k = 0;
    while (k < m && drafts[static_cast<size_t>(b) * m + k] == s_tok[k]) ++k;
    accepted_len[b] = k;
  }
}

}  // namespace

cudaError_t launch_accept(const __nv_bfloat16 *logits, const int32_t *drafts, int B, int m, int V,
                          int32_t *out_tokens, int32_t *accepted_len, cudaStream_t s) {
  if (m > kMaxRows) return cudaErrorInvalidValue;
  const int cs = m < kMaxCluster ? m : kMaxCluster;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(cs) * static_cast<unsigned>(B), 1, 1);
  cfg.blockDim = dim3(kAcceptThreads, 1, 1);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cs;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, accept_cluster_kernel, logits, drafts, m, V,
                                           out_tokens, accepted_len);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace hpd
