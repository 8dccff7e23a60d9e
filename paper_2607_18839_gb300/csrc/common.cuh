// common.cuh -- device helpers and the internal plan shared by libhpd's kernels.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/hpd.h"

namespace hpd {

constexpr int kPage = HPD_PAGE_TOKENS;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// ---------------------------------------------------------------- plan --
// Host-computed launch plan of one hpd_branch_attn call.  Only host scalars
// enter it, so it can be computed before any device data is known.
struct Plan {
  int G;           // query heads per KV head
  int rows_total;  // B * m query tokens
  int S_p;         // key splits per row tile (tcgen05: prefix + suffix blocks)
  int S_s;         // key splits of a branch's private suffix
  int tiles_max;   // upper bound of prefix row tiles per KV head
  int wr_s;        // warps along rows in the suffix kernel (1, 2, 4)
  int rt_s;        // suffix row tiles per (branch, KV head)
  bool use_tc;     // whole step on tcgen05 (G divides 128) or warp MMA stages
  bool lpt;        // tcgen05: order the units longest first (more units than SMs)
  size_t off_err;    // uint32 error word
  size_t off_ctr;    // int32 tickets [B][H_kv][rt_s]
  size_t off_opart;  // fp32 [S_p + S_s][rows_total][H_q][D]
  size_t off_lpart;  // fp32 [S_p + S_s][rows_total][H_q]
  size_t off_order;  // int32 [n_units] unit order (lpt)
  size_t bytes;      // total workspace bytes
};

// Kernel parameters of the two attention stages (prefix and suffix).
struct AttnParams {
  const __nv_bfloat16 *q;
  const __nv_bfloat16 *prefix_k;
  const __nv_bfloat16 *prefix_v;
  const int32_t *prefix_cu;
  const int32_t *branch_cu;
  const int32_t *branch_prefix_len;
  const __nv_bfloat16 *k_cache;
  const __nv_bfloat16 *v_cache;
  const int32_t *page_table;
  const int32_t *branch_len;
  const int32_t *prefix_page_table;  // [n_docs][max_prefix_pages], or null: contiguous prefix
  int max_prefix_pages;
  int n_docs, B, m, H_q, H_kv, G, D;
  int num_pages, max_pages, prefix_tokens;
  float scale_log2;  // softmax scale * log2(e)
  int S_p, S_s, rows_total;
  float *o_part;
  float *l_part;
  uint32_t *err;
  int *counters;        // per (branch, KV head, row tile) arrival tickets, zero between calls
  int *unit_ctr;        // [2] persistent-kernel unit counter and finished-CTA count, zero between calls
  int n_units;          // work units of the tcgen05 kernel (row tile x KV head x split)
  const int *unit_order;  // the order in which to take them (null: index order)
  __nv_bfloat16 *out;   // final output, written by the suffix stage
  bool out_align32;     // out is 32-byte aligned (256-bit stores)
  float *lse;           // final lse (may be null)
};

// ------------------------------------------------------- device helpers --
__device__ __forceinline__ void flag_error(uint32_t *err, uint32_t bit) {
  if (err) atomicOr(err, bit);
}

// Prefix of page d: its first token pc0 in the contiguous layout and its
// length P_d, clamped to the buffers (and, paged, to the table width); bad
// when prefix_cu is out of range (the caller flags HPD_DEVERR_PREFIX_CU).
__device__ __forceinline__ void page_prefix(const AttnParams &p, int d, int &pc0, int &P_d,
                                            bool &bad) {
  const int a0 = p.prefix_cu[d], a1 = p.prefix_cu[d + 1];
  bad = a0 < 0 || a1 < a0 || a1 > p.prefix_tokens;
  pc0 = min(max(a0, 0), p.prefix_tokens);
  P_d = min(max(a1, pc0), p.prefix_tokens) - pc0;
  if (p.prefix_page_table && P_d > p.max_prefix_pages * kPage) {
    bad = true;
    P_d = p.max_prefix_pages * kPage;
  }
}

// Pool page holding prefix page pp of page d (paged prefix); an id out of
// range is flagged and replaced by page 0.
__device__ __forceinline__ int prefix_page(const AttnParams &p, int d, int pp) {
  int pg = p.prefix_page_table[static_cast<size_t>(d) * p.max_prefix_pages + pp];
  if (pg < 0 || pg >= p.num_pages) {
    flag_error(p.err, HPD_DEVERR_PAGE_ID);
    pg = 0;
  }
  return pg;
}

// 256-bit global store of eight 32-bit words (32-byte aligned address).
__device__ __forceinline__ void st_global_v8(void *p, const uint32_t *w) {
  asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(p), "r"(w[0]),
               "r"(w[1]), "r"(w[2]), "r"(w[3]), "r"(w[4]), "r"(w[5]), "r"(w[6]), "r"(w[7])
               : "memory");
}

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// 16-byte async global->shared copy; src_bytes == 0 writes zeros.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, int src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src),
               "r"(src_bytes));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N));
}

__device__ __forceinline__ void ldmatrix_x4(uint32_t addr, uint32_t &r0, uint32_t &r1,
                                            uint32_t &r2, uint32_t &r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldmatrix_x4_trans(uint32_t addr, uint32_t &r0, uint32_t &r1,
                                                  uint32_t &r2, uint32_t &r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

// D(16x8, fp32) += A(16x16, bf16, row) * B(16x8, bf16, col)
__device__ __forceinline__ void mma_bf16_16816(float *d, const uint32_t *a, uint32_t b0,
                                               uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&v);
}

__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;\n" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ int ceil_div_i(int a, int b) { return (a + b - 1) / b; }

// Programmatic dependent launch.  A kernel launched with programmatic stream
// serialization may start while the kernel before it on the stream still
// runs; pdl_wait() returns once that kernel has finished and its writes are
// visible (at once when there is no such kernel), so everything the kernel
// reads from its predecessor comes after it.  pdl_trigger() lets the next
// such kernel start launching.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Launch `kernel`; with `overlap`, programmatically serialized after the
// previous kernel on `s` (the kernel must call pdl_wait() before using that
// kernel's results).
template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(bool overlap, void (*kernel)(KArgs...), dim3 grid, dim3 block,
                          size_t smem, cudaStream_t s, Args &&...args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = overlap ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args &&>(args)...);
}

}  // namespace hpd

// Host-side launchers (defined in the .cu files, called by hpd_api.cu).
namespace hpd {
cudaError_t launch_prefix_stage(const AttnParams &p, const Plan &plan, cudaStream_t s);
cudaError_t launch_branch_attn_tc(const AttnParams &p, const Plan &plan, bool overlap,
                                  cudaStream_t s);
cudaError_t launch_unit_order(const AttnParams &p, int tiles, int *order, cudaStream_t s);
size_t unit_order_smem_bytes(int n_docs, int B, int tiles);
cudaError_t launch_merge_splits(const AttnParams &p, bool overlap, cudaStream_t s);
cudaError_t launch_wait_selftest(uint32_t *err, uint64_t limit_ns, cudaStream_t s);
cudaError_t launch_suffix_stage(const AttnParams &p, const Plan &plan, cudaStream_t s);
// Remember `e` for hpd_last_cuda_error() and return HPD_ERR_CUDA.
hpd_status record_cuda_error(cudaError_t e);
// Every host check of an hpd_branch_attn call except the workspace's:
// scalars, required pointers and their alignment.  HPD_OK or the status the
// call would return; touches no device state.
hpd_status check_call_args(const hpd_branch_attn_args *a);
// Leading workspace bytes that must be zero before a call (error word and
// tickets); 0 if the scalars are invalid.
size_t workspace_zero_bytes(const hpd_branch_attn_args *args);
cudaError_t launch_accept(const __nv_bfloat16 *logits, const int32_t *drafts, int B, int m, int V,
                          int32_t *out_tokens, int32_t *accepted_len, cudaStream_t s);
}  // namespace hpd
