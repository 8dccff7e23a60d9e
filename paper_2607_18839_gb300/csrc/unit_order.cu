// unit_order.cu -- longest-first order of the tcgen05 kernel's work units.
//
// A unit is (row tile of 128 stacked rows, KV head, key split); its work is
// its share of the tile's key blocks: ceil(prefix keys it sees / 128) prefix
// blocks plus ceil(packed private pages / 8) suffix blocks, which depends on
// the device-side lengths.  One CTA stages the per-page and per-branch
// lengths in shared memory, computes every tile's block count there and
// writes the unit indices sorted by decreasing count (counting sort), so that
// the persistent kernel, taking units in that order, ends with its shortest
// ones (longest-processing-time-first list scheduling).  Any order gives the
// same results; only the balance across SMs changes.  Lengths are clamped as
// the attention kernel clamps them (it also flags them; this pass does not).
#include <climits>

#include "common.cuh"

namespace hpd {
namespace {

constexpr int kOrderThreads = 1024;
constexpr int kBuckets = 4 * kOrderThreads;  // block counts from kBuckets - 1 up share a bucket

// Block-wide exclusive scan of one value per thread; returns the prefix and
// adds the block total to *run (all threads).  ws: 33 ints of shared memory.
__device__ __forceinline__ int order_scan(int x, int *ws, int *run) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int incl = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int v = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += v;
  }
  if (lane == 31) ws[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const int w = ws[lane];
    int wi = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, wi, o);
      if (lane >= o) wi += v;
    }
    ws[lane] = wi - w;
    if (lane == 31) ws[32] = wi;
  }
  __syncthreads();
  const int r = *run + ws[warp] + incl - x;
  const int total = ws[32];
  __syncthreads();
  *run += total;
  return r;
}

__global__ void __launch_bounds__(kOrderThreads) unit_order_kernel(AttnParams p, int tiles,
                                                                   int *order) {
  extern __shared__ int sm[];
  __shared__ int ws[33];
  pdl_trigger();  // the attention kernel may set up meanwhile; it waits for the order
  const int nd = p.n_docs, tid = threadIdx.x;
  int *cnt = sm;                    // [kBuckets]
  int *tile_base = cnt + kBuckets;  // [nd + 1] tiles before page d
  int *c0s = tile_base + nd + 1;    // [nd] first branch of page d
  int *c1s = c0s + nd;              // [nd] one past its last branch
  int *pds = c1s + nd;              // [nd] prefix length of page d
  int *pages = pds + nd;            // [B] private pages of branch b
  int *flim = pages + p.B;          // [B] fork limit of branch b (before the page clamp)
  int *tile_n = flim + p.B;         // [tiles] key blocks of the tile
  const int m = p.m, TT = 128 / p.G;

  for (int i = tid; i < kBuckets; i += kOrderThreads) cnt[i] = 0;
  for (int b = tid; b < p.B; b += kOrderThreads) {
    const int Lb = min(max(p.branch_len[b], 0), p.max_pages * kPage);
    pages[b] = ceil_div_i(Lb, kPage);
    flim[b] = p.branch_prefix_len ? max(p.branch_prefix_len[b], 0) : INT_MAX;
  }
  int run = 0;
  for (int d0 = 0; d0 < nd; d0 += kOrderThreads) {
    const int d = d0 + tid;
    int n = 0;
    if (d < nd) {
      const int c0 = min(max(p.branch_cu[d], 0), p.B);
      const int c1 = max(min(max(p.branch_cu[d + 1], 0), p.B), c0);
      int pc0, P_d;
      bool bad;
      page_prefix(p, d, pc0, P_d, bad);
      c0s[d] = c0;
      c1s[d] = c1;
      pds[d] = P_d;
      n = ceil_div_i((c1 - c0) * m, TT);
    }
    const int before = order_scan(n, ws, &run);
    if (d < nd) tile_base[d] = before;
  }
  if (tid == 0) tile_base[nd] = run;
  __syncthreads();

  // the page owning tile t: the last d with tile_base[d] <= t (it has tiles)
  for (int t = tid; t < tiles; t += kOrderThreads) {
    int N = 0;
    if (t < tile_base[nd]) {
      int lo = 0, hi = nd;
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (tile_base[mid] <= t) lo = mid; else hi = mid;
      }
      const int d = lo, lt = t - tile_base[d], b0 = c0s[d], b1 = c1s[d], P_d = pds[d];
      const int tok0 = b0 * m + lt * TT;
      const int ntok = min(TT, (b1 - b0) * m - lt * TT);
      const int b_lo = tok0 / m;
      const int nbc = (tok0 + ntok - 1) / m - b_lo + 1;
      int np = 0, kmax = 0;
      for (int bl = 0; bl < nbc; ++bl) {
        np += pages[b_lo + bl];
        kmax = max(kmax, min(flim[b_lo + bl], P_d));
      }
      N = ceil_div_i(kmax, 128) + ceil_div_i(np, 128 / kPage);
    }
    tile_n[t] = N;
  }
  __syncthreads();

  // unit u = (tile * H_kv + g) * S_p + split takes blocks
  // [split N / S_p, (split + 1) N / S_p) of its tile; bucket by descending count
  auto key_of = [&](int u) {
    const int split = u % p.S_p, tile = u / (p.S_p * p.H_kv);
    const long long N = tile_n[tile];
    const int n = static_cast<int>((split + 1) * N / p.S_p - split * N / p.S_p);
    return kBuckets - 1 - min(n, kBuckets - 1);  // 0: the longest
  };
  for (int u = tid; u < p.n_units; u += kOrderThreads) atomicAdd(&cnt[key_of(u)], 1);
  __syncthreads();
  // exclusive prefix over the buckets, kBuckets / kOrderThreads per thread
  int c[kBuckets / kOrderThreads], own = 0;
#pragma unroll
  for (int i = 0; i < kBuckets / kOrderThreads; ++i) {
    c[i] = cnt[tid * (kBuckets / kOrderThreads) + i];
    own += c[i];
  }
  int zero = 0;
  int pos = order_scan(own, ws, &zero);
#pragma unroll
  for (int i = 0; i < kBuckets / kOrderThreads; ++i) {
    cnt[tid * (kBuckets / kOrderThreads) + i] = pos;
    pos += c[i];
  }
  __syncthreads();
  for (int u = tid; u < p.n_units; u += kOrderThreads) order[atomicAdd(&cnt[key_of(u)], 1)] = u;
}

}  // namespace

size_t unit_order_smem_bytes(int n_docs, int B, int tiles) {
  return sizeof(int) * (static_cast<size_t>(kBuckets) + 4 * static_cast<size_t>(n_docs) + 1 +
                        2 * static_cast<size_t>(B) + static_cast<size_t>(tiles));
}

cudaError_t launch_unit_order(const AttnParams &p, int tiles, int *order, cudaStream_t s) {
  const size_t smem = unit_order_smem_bytes(p.n_docs, p.B, tiles);
  if (smem > 48 * 1024) {
    const cudaError_t e = cudaFuncSetAttribute(
        unit_order_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  unit_order_kernel<<<1, kOrderThreads, smem, s>>>(p, tiles, order);
  return cudaGetLastError();
}

}  // namespace hpd
