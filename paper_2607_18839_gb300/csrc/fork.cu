// fork.cu -- fork detection and child branches after verification
// (Algorithm 1: scan the accepted tokens for the fork token and spawn a
// child that shares the parent's context; Sec. 3.3 "Dynamic Branch Forking").
//
// The shared context of a page is its prefix (vision tokens, then the layout
// branch's tokens), so a child is a new branch of the same page whose
// fork-position prefix length is the position just past the fork token, with
// no private keys yet: nothing is copied, the prefix keys are shared.
//
// A layout branch b emits t*_{b,0..e_b-1}, e_b = min(n_acc_b + 1, m) (the
// accepted drafts and the correction token); the token at index i sits at
// prefix position layout_pos[b] + i.  Every emitted fork token spawns one
// child with prefix length layout_pos[b] + i + 1.  The new branch arrays keep
// each page's old branches in order and append its children after them, in
// (parent, index) order; the placement comes from a scan in branch order, so
// it is deterministic.
//
// One launch (B + n_docs up to kMaxFused): every CTA counts every branch's
// children and scans the counts in its own shared memory (the outputs never
// alias the inputs, so no CTA waits for another), then writes its share of
// the new arrays.  With c_b the children of branch b and pre_b their
// exclusive sum over branches, page d's old branches move by pre at its first
// branch, and branch b's children start at new index branch_cu[d+1] + pre_b.
// Larger calls take two launches (one CTA scans page by page, then many copy).
#include <algorithm>

#include "common.cuh"

namespace hpd {
namespace {

constexpr int kForkThreads = 1024;
constexpr int kFusedThreads = 256;
constexpr int kMaxFused = 12000;  // B + n_docs + 2 ints of shared memory (48,000 bytes)

// Block-wide exclusive scan of one value per thread; total to *total.
__device__ __forceinline__ int fork_scan(int x, int *ws, int *total) {
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
    const int w = lane < kForkThreads / 32 ? ws[lane] : 0;
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
  const int r = ws[warp] + incl - x;
  *total = ws[32];
  __syncthreads();
  return r;
}

__device__ __forceinline__ int n_forks(const hpd_fork_args &a, int b) {
  if (a.is_layout && !a.is_layout[b]) return 0;
  const int n = a.accepted_len[b];
  const int e = n < 0 ? 0 : min(n + 1, a.m);
  int f = 0;
  for (int i = 0; i < e; ++i) f += a.out_tokens[static_cast<size_t>(b) * a.m + i] == a.fork_token;
  return f;
}

// page of branch b (branch_cu was validated at the start of the kernel)
__device__ __forceinline__ int doc_of(const hpd_fork_args &a, int b) {
  int lo = 0, hi = a.n_docs;  // largest d with branch_cu[d] <= b
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (a.branch_cu[mid] <= b) lo = mid; else hi = mid;
  }
  return lo;
}

__global__ void __launch_bounds__(kForkThreads) fork_kernel(hpd_fork_args a) {
  __shared__ int ws[33];
  __shared__ int s_total, s_bad;
  uint32_t *err = static_cast<uint32_t *>(a.workspace);
  int *doc_base = static_cast<int *>(a.workspace) + 64;  // [n_docs + 1] children before doc d
  const int tid = threadIdx.x;
  if (tid == 0) {
    s_total = 0;
    s_bad = a.branch_cu[0] != 0 || a.branch_cu[a.n_docs] != a.B;
  }
  __syncthreads();
  for (int d = tid; d < a.n_docs; d += kForkThreads)
    if (a.branch_cu[d] > a.branch_cu[d + 1]) s_bad = 1;
  __syncthreads();
  int *ok_word = static_cast<int *>(a.workspace) + 1;  // read by fork_copy_kernel
  if (s_bad) {  // nothing written but the error
    if (tid == 0) {
      atomicOr(err, HPD_DEVERR_BRANCH_CU);
      *a.new_B = -1;
      *ok_word = 0;
    }
    return;
  }
  // children per page, exclusive over pages
  for (int d0 = 0; d0 < a.n_docs; d0 += kForkThreads) {
    const int d = d0 + tid;
    int c = 0;
    if (d < a.n_docs)
      for (int b = a.branch_cu[d]; b < a.branch_cu[d + 1]; ++b) c += n_forks(a, b);
    int total;
    const int before = fork_scan(c, ws, &total);
    if (d < a.n_docs) doc_base[d] = s_total + before;
    __syncthreads();
    if (tid == 0) s_total += total;
    __syncthreads();
  }
  const int n_children = s_total;
  if (a.B + n_children > a.cap) {
    if (tid == 0) {
      atomicOr(err, HPD_DEVERR_FORK_CAP);
      *a.new_B = -1;
      *ok_word = 0;
    }
    return;
  }
  if (tid == 0) {
    doc_base[a.n_docs] = n_children;
    *a.new_B = a.B + n_children;
    *ok_word = 1;
  }
  __syncthreads();
  for (int d = tid; d <= a.n_docs; d += kForkThreads) a.new_branch_cu[d] = a.branch_cu[d] + doc_base[d];
  // children: after their page's old branches, in (parent, index) order
  int base = 0;
  for (int b0 = 0; b0 < a.B; b0 += kForkThreads) {
    const int b = b0 + tid;
    const int f = b < a.B ? n_forks(a, b) : 0;
    int total;
    const int before = fork_scan(f, ws, &total);  // children of branches < b (all pages)
    if (f > 0) {
      const int d = doc_of(a, b);
      // children of earlier pages come before this page's, and sit in earlier
      // pages' ranges; subtract them to index within the page
      int slot = a.branch_cu[d + 1] + doc_base[d] + (base + before - doc_base[d]);
      const int n = a.accepted_len[b];
      const int e = n < 0 ? 0 : min(n + 1, a.m);
      for (int i = 0; i < e; ++i) {
        if (a.out_tokens[static_cast<size_t>(b) * a.m + i] != a.fork_token) continue;
        a.new_parent[slot] = -1 - b;  // a child of b
        a.new_branch_len[slot] = 0;
        a.new_branch_prefix_len[slot] = a.layout_pos[b] + i + 1;
        for (int pgi = 0; pgi < a.max_pages; ++pgi)
          a.new_page_table[static_cast<size_t>(slot) * a.max_pages + pgi] = -1;
        ++slot;
      }
    }
    base += total;
  }
}

// The whole fork step in one launch (see the top of the file).
__global__ void __launch_bounds__(kFusedThreads) fork_fused_kernel(hpd_fork_args a) {
  extern __shared__ int s_dyn[];
  int *pre = s_dyn;                 // [B + 1] children of branches before b
  int *cu = s_dyn + a.B + 1;        // [n_docs + 1] branch_cu
  __shared__ int warp_sums[kFusedThreads / 32];
  __shared__ int s_bad, s_total;
  uint32_t *err = static_cast<uint32_t *>(a.workspace);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  pdl_wait();  // whatever ran before on the stream has finished
  if (tid == 0) {
    s_bad = a.branch_cu[0] != 0 || a.branch_cu[a.n_docs] != a.B;
    s_total = 0;
  }
  for (int d = tid; d <= a.n_docs; d += kFusedThreads) cu[d] = a.branch_cu[d];
  __syncthreads();
  for (int d = tid; d < a.n_docs; d += kFusedThreads)
    if (cu[d] > cu[d + 1]) s_bad = 1;
  __syncthreads();
  if (s_bad) {  // nothing written but the error
    if (blockIdx.x == 0 && tid == 0) {
      atomicOr(err, HPD_DEVERR_BRANCH_CU);
      *a.new_B = -1;
    }
    return;
  }
  for (int b0 = 0; b0 < a.B; b0 += kFusedThreads) {
    const int b = b0 + tid;
    const int f = b < a.B ? n_forks(a, b) : 0;
    int incl = f;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    if (lane == 31) warp_sums[warp] = incl;
    __syncthreads();
    int woff = 0;
    for (int w = 0; w < warp; ++w) woff += warp_sums[w];
    if (b < a.B) pre[b] = s_total + woff + incl - f;
    __syncthreads();
    if (tid == kFusedThreads - 1) s_total += woff + incl;
    __syncthreads();
  }
  if (tid == 0) pre[a.B] = s_total;
  __syncthreads();
  const int n_children = s_total;
  if (a.B + n_children > a.cap) {
    if (blockIdx.x == 0 && tid == 0) {
      atomicOr(err, HPD_DEVERR_FORK_CAP);
      *a.new_B = -1;
    }
    return;
  }
  // page of branch b: the largest d with cu[d] <= b
  auto doc = [&](int b) {
    int lo = 0, hi = a.n_docs;
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (cu[mid] <= b) lo = mid; else hi = mid;
    }
    return lo;
  };
  const size_t stride = static_cast<size_t>(gridDim.x) * kFusedThreads;
  const size_t t0 = static_cast<size_t>(blockIdx.x) * kFusedThreads + tid;
  if (t0 == 0) *a.new_B = a.B + n_children;
  for (size_t d = t0; d <= static_cast<size_t>(a.n_docs); d += stride)
    a.new_branch_cu[d] = cu[d] + pre[cu[d]];
  for (size_t b = t0; b < static_cast<size_t>(a.B); b += stride) {
    const int ib = static_cast<int>(b), d = doc(ib);
    const size_t nb = b + pre[cu[d]];
    a.new_parent[nb] = ib;
    a.new_branch_len[nb] = a.branch_len[b];
    a.new_branch_prefix_len[nb] = a.branch_prefix_len ? a.branch_prefix_len[b] : -1;
    const int f = pre[ib + 1] - pre[ib];
    if (f > 0) {  // its children: after the page's old branches, in index order
      int slot = cu[d + 1] + pre[ib];
      const int n = a.accepted_len[b];
      const int e = n < 0 ? 0 : min(n + 1, a.m);
      for (int i = 0; i < e; ++i) {
        if (a.out_tokens[b * a.m + i] != a.fork_token) continue;
        a.new_parent[slot] = -1 - ib;
        a.new_branch_len[slot] = 0;
        a.new_branch_prefix_len[slot] = a.layout_pos[b] + i + 1;
        ++slot;
      }
    }
  }
  for (size_t i = t0; i < static_cast<size_t>(a.B) * a.max_pages; i += stride) {
    const int b = static_cast<int>(i / a.max_pages);
    const size_t nb = b + pre[cu[doc(b)]];
    a.new_page_table[nb * a.max_pages + i % a.max_pages] = a.page_table[i];
  }
  // the children's page-table rows are all -1
  for (size_t i = t0; i < static_cast<size_t>(n_children) * a.max_pages; i += stride) {
    // child number c (in new-index order over pages) -> its new index
    const int c = static_cast<int>(i / a.max_pages);
    int lo = 0, hi = a.n_docs;  // the page holding child c: largest d with pre[cu[d]] <= c
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (pre[cu[mid]] <= c) lo = mid; else hi = mid;
    }
    const size_t slot = cu[lo + 1] + c;  // children of page lo after its old branches
    a.new_page_table[slot * a.max_pages + i % a.max_pages] = -1;
  }
}

// The old branches' arrays, moved past the children of earlier pages (many
// CTAs, after fork_kernel on the same stream; nothing when it failed).
__global__ void fork_copy_kernel(hpd_fork_args a) {
  if (*reinterpret_cast<volatile int *>(static_cast<int *>(a.workspace) + 1) == 0) return;
  const int *doc_base = static_cast<const int *>(a.workspace) + 64;
  const size_t stride = static_cast<size_t>(gridDim.x) * blockDim.x;
  const size_t t0 = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  for (size_t b = t0; b < static_cast<size_t>(a.B); b += stride) {
    const size_t nb = b + doc_base[doc_of(a, static_cast<int>(b))];
    a.new_parent[nb] = static_cast<int>(b);
    a.new_branch_len[nb] = a.branch_len[b];
    a.new_branch_prefix_len[nb] = a.branch_prefix_len ? a.branch_prefix_len[b] : -1;
  }
  for (size_t i = t0; i < static_cast<size_t>(a.B) * a.max_pages; i += stride) {
    const int b = static_cast<int>(i / a.max_pages);
    const size_t nb = b + doc_base[doc_of(a, b)];
    a.new_page_table[nb * a.max_pages + i % a.max_pages] = a.page_table[i];
  }
}

}  // namespace
}  // namespace hpd

extern "C" hpd_status hpd_fork_children(const hpd_fork_args *a, hpd_stream_t stream) {
  if (!a || !a->branch_cu || !a->new_branch_cu || !a->new_B || !a->workspace)
    return HPD_ERR_INVALID_ARG;
  // per-branch arrays may be null only when there are no branches at all
  if (a->B > 0 && (!a->out_tokens || !a->accepted_len || !a->layout_pos || !a->branch_len ||
                   !a->page_table || !a->new_branch_prefix_len || !a->new_branch_len ||
                   !a->new_page_table || !a->new_parent))
    return HPD_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(a->workspace) & 255u) != 0) return HPD_ERR_WORKSPACE;
  if (a->B < 0 || a->m < 1 || a->m > 64 || a->n_docs < 1 || a->max_pages < 1 || a->cap < a->B)
    return HPD_ERR_INVALID_ARG;
  if (a->workspace_bytes < static_cast<size_t>(64 + a->n_docs + 1) * sizeof(int))
    return HPD_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = cudaSuccess;
  if (static_cast<long long>(a->B) + a->n_docs + 2 <= hpd::kMaxFused) {
    // one launch; it may start while the previous kernel on the stream
    // finishes (it waits for it before reading anything)
    const long long n = static_cast<long long>(a->B) * a->max_pages;
    const int grid = static_cast<int>(std::max<long long>(1, std::min<long long>((n + 2047) / 2048, 64)));
    const size_t smem = sizeof(int) * (static_cast<size_t>(a->B) + a->n_docs + 2);
    e = hpd::launch_kernel(true, hpd::fork_fused_kernel, dim3(grid), dim3(hpd::kFusedThreads), smem,
                           s, *a);
  } else {
    hpd::fork_kernel<<<1, hpd::kForkThreads, 0, s>>>(*a);
    if (a->B > 0) {
      const long long n = static_cast<long long>(a->B) * a->max_pages;
      const int grid = static_cast<int>(std::min<long long>((n + 255) / 256, 1216));
      hpd::fork_copy_kernel<<<grid, 256, 0, s>>>(*a);
    }
    e = cudaGetLastError();
  }
  return e == cudaSuccess ? HPD_OK : hpd::record_cuda_error(e);
}
