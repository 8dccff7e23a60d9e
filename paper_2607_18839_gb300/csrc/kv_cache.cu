// kv_cache.cu -- paged private KV around a decode step (Algorithm 1: the
// step's tokens are written to the cache before attention, and after the
// verification the branch keeps only what was accepted).
//
//   hpd_kv_append    branch b's m new K/V rows go to private positions
//                    [L_b, L_b + m); the logical pages this opens are taken
//                    from a device stack of free page ids; L_b += m.
//   hpd_kv_rollback  the step's m positions [L_b - m, L_b) keep their first
//                    keep_b = min(n_acc_b + 1, m) rows (0 when n_acc_b < 0);
//                    L_b -= m - keep_b, and the logical pages that no longer
//                    hold a row go back onto the stack (table entry -1).
//
// Allocation is deterministic: one CTA scans the per-branch page counts in
// branch order, so branch b takes (or returns) the stack entries right after
// those of branches 0..b-1, whatever the launch order.  All or nothing: when
// the stack is short or a branch would outgrow its table row, nothing
// changes and the error word gets HPD_DEVERR_POOL / HPD_DEVERR_BRANCH_LEN.
// Up to kScanThreads branches the scan is one pass (each thread keeps its
// branch's values); beyond, a first pass checks the capacity and a second
// assigns.  Each kernel is launched with programmatic dependent launch: it
// waits for its predecessor on the stream before touching any state, and
// lets its successor start launching right away.
#include <algorithm>

#include "common.cuh"

namespace hpd {
namespace {

constexpr int kScanThreads = 1024;

// The C ABI arguments with the workspace words resolved.
struct KvArgs {
  const void *k_new, *v_new;
  void *k_cache, *v_cache;
  int32_t *page_table, *branch_len, *free_pages, *free_top;
  uint32_t *err;   // workspace word 0: HPD_DEVERR_* bits
  int32_t *done;   // workspace word 1: 1 when the last append allocated
  int B, m, H_kv, D, num_pages, max_pages;
};

__device__ __forceinline__ int pages_of(int len) { return (len + kPage - 1) / kPage; }

// Block-wide exclusive scan of one value per thread; returns the prefix and
// writes the block total to *total (every thread).
__device__ __forceinline__ int block_scan(int x, int *warp_sums, int *total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int incl = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int v = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += v;
  }
  if (lane == 31) warp_sums[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    int w = lane < kScanThreads / 32 ? warp_sums[lane] : 0;
    int wi = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, wi, o);
      if (lane >= o) wi += v;
    }
    warp_sums[lane] = wi - w;  // exclusive warp offsets
    if (lane == 31) warp_sums[32] = wi;
  }
  __syncthreads();
  const int r = warp_sums[warp] + incl - x;
  *total = warp_sums[32];
  __syncthreads();  // warp_sums is reused by the next call
  return r;
}

// Pass 1 of the append (one CTA): check capacity, take page ids, extend the
// lengths.  Branches are walked in chunks of kScanThreads.
__global__ void __launch_bounds__(kScanThreads) kv_append_alloc_kernel(KvArgs a) {
  __shared__ int warp_sums[33];
  __shared__ int s_bad, s_need;
  const int tid = threadIdx.x;
  pdl_wait();     // the previous kernel's lengths, tables and stack
  pdl_trigger();  // the copy may launch; it waits for this kernel
  if (tid == 0) {
    s_bad = 0;
    s_need = 0;
  }
  __syncthreads();
  if (a.B <= kScanThreads) {  // one pass
    const int b = tid;
    int need = 0, L = 0;
    if (b < a.B) {
      L = a.branch_len[b];
      if (L < 0 || L + a.m > a.max_pages * kPage) atomicOr(&s_bad, 1);
      else need = pages_of(L + a.m) - pages_of(L);
    }
    int total;
    const int before = block_scan(need, warp_sums, &total);  // orders the s_bad writes
    const int top = *a.free_top;
    if (s_bad || total > top || top > a.num_pages) {
      if (tid == 0) {
        atomicOr(a.err, s_bad ? HPD_DEVERR_BRANCH_LEN : HPD_DEVERR_POOL);
        *a.done = 0;
      }
      return;
    }
    if (b < a.B) {
      int32_t *row = a.page_table + static_cast<size_t>(b) * a.max_pages;
      for (int i = 0; i < need; ++i) row[pages_of(L) + i] = a.free_pages[top - total + before + i];
      a.branch_len[b] = L + a.m;
    }
    if (tid == 0) {
      *a.free_top = top - total;
      *a.done = 1;
    }
    return;
  }
  // capacity check and total pages needed
  for (int b0 = 0; b0 < a.B; b0 += kScanThreads) {
    const int b = b0 + tid;
    int need = 0;
    if (b < a.B) {
      const int L = a.branch_len[b];
      if (L < 0 || L + a.m > a.max_pages * kPage) atomicOr(&s_bad, 1);
      else need = pages_of(L + a.m) - pages_of(L);
    }
    int total;
    block_scan(need, warp_sums, &total);
    if (tid == 0) s_need += total;
    __syncthreads();
  }
  const int top = *a.free_top;
  if (s_bad || s_need > top || top > a.num_pages) {
    if (tid == 0) {
      atomicOr(a.err, s_bad ? HPD_DEVERR_BRANCH_LEN : HPD_DEVERR_POOL);
      *a.done = 0;
    }
    return;
  }
  // branch b takes stack entries [top - need_all + before_b, ...)
  int base = top - s_need;
  for (int b0 = 0; b0 < a.B; b0 += kScanThreads) {
    const int b = b0 + tid;
    int need = 0, L = 0;
    if (b < a.B) {
      L = a.branch_len[b];
      need = pages_of(L + a.m) - pages_of(L);
    }
    int total;
    const int before = block_scan(need, warp_sums, &total);
    if (b < a.B) {
      int32_t *row = a.page_table + static_cast<size_t>(b) * a.max_pages;
      for (int i = 0; i < need; ++i) row[pages_of(L) + i] = a.free_pages[base + before + i];
      a.branch_len[b] = L + a.m;
    }
    base += total;
  }
  __syncthreads();
  if (tid == 0) {
    *a.free_top = top - s_need;
    *a.done = 1;
  }
}

// Pass 2 of the append: copy the new rows, 16 bytes per thread, when pass 1
// succeeded (*done; otherwise nothing was allocated and nothing is written).
__global__ void kv_append_copy_kernel(KvArgs a, int rows_total) {
  pdl_wait();  // the allocation
  pdl_trigger();
  if (*reinterpret_cast<volatile int32_t *>(a.done) == 0) return;
  const int vec_per_row = a.D / 8;  // 16-byte vectors of one (row, head)
  const long long n = static_cast<long long>(rows_total) * a.H_kv * vec_per_row;
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int v = static_cast<int>(i % vec_per_row);
    const long long rh = i / vec_per_row;
    const int hh = static_cast<int>(rh % a.H_kv);
    const int r = static_cast<int>(rh / a.H_kv);  // b * m + j
    const int b = r / a.m, j = r % a.m;
    const int pos = a.branch_len[b] - a.m + j;    // length already extended
    if (pos < 0 || pos >= a.max_pages * kPage) continue;
    const int pg = a.page_table[static_cast<size_t>(b) * a.max_pages + pos / kPage];
    if (pg < 0 || pg >= a.num_pages) continue;
    const size_t src = (static_cast<size_t>(r) * a.H_kv + hh) * a.D / 8 + v;
    const size_t dst = ((static_cast<size_t>(pg) * kPage + pos % kPage) * a.H_kv + hh) * a.D / 8 + v;
    reinterpret_cast<uint4 *>(a.k_cache)[dst] = reinterpret_cast<const uint4 *>(a.k_new)[src];
    reinterpret_cast<uint4 *>(a.v_cache)[dst] = reinterpret_cast<const uint4 *>(a.v_new)[src];
  }
}

// Rollback (one CTA): keep the first keep_b of the step's m rows, free the
// logical pages past the new length, push their ids in branch order.
__global__ void __launch_bounds__(kScanThreads)
    kv_rollback_kernel(KvArgs a, const int32_t *__restrict__ accepted_len) {
  __shared__ int warp_sums[33];
  __shared__ int s_bad, s_free;
  const int tid = threadIdx.x;
  pdl_wait();  // the previous kernel's lengths, tables, stack and accepted lengths
  pdl_trigger();
  if (tid == 0) {
    s_bad = 0;
    s_free = 0;
  }
  __syncthreads();
  auto new_len = [&](int b, int L) {
    const int n = accepted_len[b];
    const int keep = n < 0 ? 0 : min(n + 1, a.m);
    return L - a.m + keep;
  };
  if (a.B <= kScanThreads) {  // one pass
    const int b = tid;
    int fr = 0, L = 0, Ln = 0;
    if (b < a.B) {
      L = a.branch_len[b];
      if (L < a.m || L > a.max_pages * kPage) {
        atomicOr(&s_bad, 1);
      } else {
        Ln = new_len(b, L);
        fr = pages_of(L) - pages_of(Ln);
      }
    }
    int total;
    const int before = block_scan(fr, warp_sums, &total);  // orders the s_bad writes
    const int top = *a.free_top;
    if (s_bad || top < 0 || top + total > a.num_pages) {
      if (tid == 0) atomicOr(a.err, s_bad ? HPD_DEVERR_BRANCH_LEN : HPD_DEVERR_POOL);
      return;
    }
    if (b < a.B) {
      int32_t *row = a.page_table + static_cast<size_t>(b) * a.max_pages;
      for (int i = 0; i < fr; ++i) {
        a.free_pages[top + before + i] = row[pages_of(Ln) + i];
        row[pages_of(Ln) + i] = -1;
      }
      a.branch_len[b] = Ln;
    }
    if (tid == 0) *a.free_top = top + total;
    return;
  }
  for (int b0 = 0; b0 < a.B; b0 += kScanThreads) {
    const int b = b0 + tid;
    int fr = 0;
    if (b < a.B) {
      const int L = a.branch_len[b];
      if (L < a.m || L > a.max_pages * kPage) atomicOr(&s_bad, 1);
      else fr = pages_of(L) - pages_of(new_len(b, L));
    }
    int total;
    block_scan(fr, warp_sums, &total);
    if (tid == 0) s_free += total;
    __syncthreads();
  }
  const int top = *a.free_top;
  if (s_bad || top < 0 || top + s_free > a.num_pages) {
    if (tid == 0) atomicOr(a.err, s_bad ? HPD_DEVERR_BRANCH_LEN : HPD_DEVERR_POOL);
    return;
  }
  int base = top;
  for (int b0 = 0; b0 < a.B; b0 += kScanThreads) {
    const int b = b0 + tid;
    int fr = 0, L = 0, Ln = 0;
    if (b < a.B) {
      L = a.branch_len[b];
      Ln = new_len(b, L);
      fr = pages_of(L) - pages_of(Ln);
    }
    int total;
    const int before = block_scan(fr, warp_sums, &total);
    if (b < a.B) {
      int32_t *row = a.page_table + static_cast<size_t>(b) * a.max_pages;
      for (int i = 0; i < fr; ++i) {
        a.free_pages[base + before + i] = row[pages_of(Ln) + i];
        row[pages_of(Ln) + i] = -1;
      }
      a.branch_len[b] = Ln;
    }
    base += total;
  }
  __syncthreads();
  if (tid == 0) *a.free_top = top + s_free;
}

}  // namespace

// ------------------------------------------------------------------ C ABI --
namespace {

hpd_status kv_check(const hpd_kv_args *a, KvArgs *k) {
  if (!a || !a->k_cache || !a->v_cache || !a->page_table || !a->branch_len ||
      !a->free_pages || !a->free_top || !a->workspace)
    return HPD_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(a->workspace) & 255u) != 0) return HPD_ERR_WORKSPACE;
  if (a->B < 0 || a->m < 1 || a->m > 64 || a->H_kv < 1 || (a->D != 64 && a->D != 128) ||
      a->num_pages < 1 || a->max_pages < 1)
    return HPD_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(a->k_cache) | reinterpret_cast<uintptr_t>(a->v_cache)) & 15u)
    return HPD_ERR_INVALID_ARG;
  *k = KvArgs{a->k_new, a->v_new, a->k_cache, a->v_cache, a->page_table, a->branch_len,
              a->free_pages, a->free_top, static_cast<uint32_t *>(a->workspace),
              static_cast<int32_t *>(a->workspace) + 1, a->B, a->m, a->H_kv, a->D,
              a->num_pages, a->max_pages};
  return HPD_OK;
}

}  // namespace
}  // namespace hpd

extern "C" {

hpd_status hpd_kv_append(const hpd_kv_args *args, hpd_stream_t stream) {
  hpd::KvArgs k;
  const hpd_status st = hpd::kv_check(args, &k);
  if (st != HPD_OK) return st;
  if (!args->k_new || !args->v_new ||
      ((reinterpret_cast<uintptr_t>(args->k_new) | reinterpret_cast<uintptr_t>(args->v_new)) & 15u))
    return HPD_ERR_INVALID_ARG;
  if (args->B == 0) return HPD_OK;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = hpd::launch_kernel(true, hpd::kv_append_alloc_kernel, dim3(1),
                                     dim3(hpd::kScanThreads), 0, s, k);
  const long long vecs = static_cast<long long>(args->B) * args->m * args->H_kv * (args->D / 8);
  const int grid = static_cast<int>(std::min<long long>((vecs + 255) / 256, 152 * 8));
  if (e == cudaSuccess)
    e = hpd::launch_kernel(true, hpd::kv_append_copy_kernel, dim3(grid), dim3(256), 0, s, k,
                           args->B * args->m);
  return e == cudaSuccess ? HPD_OK : hpd::record_cuda_error(e);
}

hpd_status hpd_kv_rollback(const hpd_kv_args *args, const int32_t *accepted_len,
                           hpd_stream_t stream) {
  hpd::KvArgs k;
  const hpd_status st = hpd::kv_check(args, &k);
  if (st != HPD_OK) return st;
  if (!accepted_len) return HPD_ERR_INVALID_ARG;
  if (args->B == 0) return HPD_OK;
  const cudaError_t e =
      hpd::launch_kernel(true, hpd::kv_rollback_kernel, dim3(1), dim3(hpd::kScanThreads), 0,
                         reinterpret_cast<cudaStream_t>(stream), k, accepted_len);
  return e == cudaSuccess ? HPD_OK : hpd::record_cuda_error(e);
}

}  // extern "C"
