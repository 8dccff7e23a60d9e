// hpd_api.cu -- the C ABI of libhpd (include/hpd.h): host-side validation,
// the launch plan and the workspace layout.  Every compute step runs in the
// kernels of branch_attn_tc.cu, merge.cu, attn_mma.cu and accept.cu; nothing
// here touches device data.
#include <cmath>
#include <cstdint>
#include <mutex>

#include "common.cuh"

namespace {

thread_local int g_last_cuda_error = 0;

hpd_status cuda_fail(cudaError_t e) {
  g_last_cuda_error = static_cast<int>(e);
  return HPD_ERR_CUDA;
}

constexpr size_t kAlign = 256;
constexpr int kPrefixTileRows = 64;   // rows per prefix-stage CTA
constexpr int kPlanSms = 152;          // SMs the split plan assumes (GB300)
constexpr int kTargetCtas = kPlanSms * 4;  // warp-MMA prefix CTAs aimed for
constexpr int kTcTileRows = 128;       // stacked rows of one tcgen05 prefix CTA
constexpr int kMaxPrefixSplits = 8;
constexpr int kLptWaves = 2;
constexpr double kLptMinUs = 250.0;
constexpr size_t kOrderSmemMax = 200 * 1024;
constexpr int kSuffixSplitKeys = 1536;  // a suffix chunk holds at most ~this many keys
constexpr int kMaxSuffixSplits = 8;

size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }
int ceil_div(long long a, long long b) { return static_cast<int>((a + b - 1) / b); }
bool aligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Host-scalar checks shared by the workspace query and the call itself.
hpd_status check_scalars(const hpd_branch_attn_args *a) {
  if (!a) return HPD_ERR_INVALID_ARG;
  if (a->n_docs < 1 || a->B < 1 || a->m < 1 || a->H_q < 1 || a->H_kv < 1 || a->num_pages < 1 ||
      a->max_pages_per_branch < 1 || a->prefix_tokens < 0 || a->max_prefix_len < 0)
    return HPD_ERR_INVALID_ARG;
  if (a->prefix_page_table && a->max_prefix_pages < 1) return HPD_ERR_INVALID_ARG;
  if (a->m > 16) return HPD_ERR_UNSUPPORTED;
  if (a->H_q % a->H_kv != 0) return HPD_ERR_INVALID_ARG;
  if (a->H_q / a->H_kv > 16) return HPD_ERR_UNSUPPORTED;
  if (a->D != 64 && a->D != 128) return HPD_ERR_UNSUPPORTED;
  if (!std::isfinite(a->scale)) return HPD_ERR_INVALID_ARG;
  const long long rows = static_cast<long long>(a->B) * a->m;
  if (rows * a->H_q * a->D >= (1LL << 31)) return HPD_ERR_UNSUPPORTED;
  if (static_cast<long long>(a->max_pages_per_branch) * hpd::kPage >= (1LL << 30))
    return HPD_ERR_UNSUPPORTED;
  return HPD_OK;
}

hpd::Plan make_plan(const hpd_branch_attn_args *a) {
  hpd::Plan pl{};
  pl.G = a->H_q / a->H_kv;
  pl.rows_total = a->B * a->m;
  int maxP = a->max_prefix_len > 0 ? std::min(a->max_prefix_len, a->prefix_tokens)
                                   : a->prefix_tokens;
  if (a->prefix_page_table)
    maxP = static_cast<int>(std::min<long long>(maxP, 16LL * a->max_prefix_pages));
  pl.use_tc = (a->D == 64 || a->D == 128) && (kTcTileRows % pl.G == 0);
  if (pl.use_tc) {
    // tcgen05 kernel: units of 128 stacked rows (128 / G tokens) of one
    // page and KV head, one CTA per SM taking units in turn.
    const int tile_tokens = kTcTileRows / pl.G;
    const int tiles = ceil_div(static_cast<long long>(a->B) * a->m, tile_tokens);
    pl.tiles_max = tiles + a->n_docs;
    // Key splits: minimise the estimated time of the step, i.e. waves of
    // CTAs x (blocks per CTA + 1 for prologue / epilogue) x time per block,
    // plus, when split, the merge launch and its partial-result traffic.
    // A CTA walks its page's prefix blocks and its branches' private pages
    // (guessed at a quarter of the page-table width per branch).
    const long long ctas = static_cast<long long>(std::max(tiles, 1)) * a->H_kv;
    const int branches_per_cta =
        std::max(1, kTcTileRows / std::max(1, a->m * pl.G));
    const int nb = std::max(1, ceil_div(maxP, 128)) +
                   ceil_div(static_cast<long long>(branches_per_cta) *
                                std::max(1, a->max_pages_per_branch / 4), 8);
    const double block_us = 0.7;  // one 128-key block, measured order
    const double partial_bytes =
        static_cast<double>(a->B) * a->m * a->H_q * (a->D + 1) * sizeof(float);
    int best = 1;
    double best_cost = -1.0;
    for (int sp = 1; sp <= std::min(nb, kMaxPrefixSplits); ++sp) {
      const long long waves = (ctas * sp + kPlanSms - 1) / kPlanSms;
      double cost = static_cast<double>(waves) * (ceil_div(nb, sp) + 1) * block_us;
      if (sp > 1) cost += 4.0 + sp * partial_bytes / 4.0e6;  // ~4 TB/s
      if (best_cost < 0 || cost < best_cost) {
        best_cost = cost;
        best = sp;
      }
    }
    pl.S_p = best;
    // With at least kLptWaves units per SM, units of unequal length leave
    // SMs idle at the end; a one-CTA pass then orders them longest first
    // (it holds the per-page and per-branch lengths in shared memory).  The
    // pass costs about 10 us and saves a few percent of the kernel, so it
    // runs only when the kernel is estimated at kLptMinUs or more.
    const double est_us = static_cast<double>(ctas) * best * (ceil_div(nb, best) + 1) *
                          block_us / kPlanSms;
    pl.lpt = ctas * best >= kLptWaves * kPlanSms && est_us >= kLptMinUs &&
             hpd::unit_order_smem_bytes(a->n_docs, a->B, pl.tiles_max) <= kOrderSmemMax;
  } else {
    const long long stacked = static_cast<long long>(a->B) * a->m * pl.G;
    const int tiles = ceil_div(stacked, kPrefixTileRows);
    pl.tiles_max = tiles + a->n_docs;
    const long long tiles_est = static_cast<long long>(std::max(tiles, 1)) * a->H_kv;
    int sp = ceil_div(kTargetCtas, tiles_est);
    sp = std::min(sp, std::max(1, ceil_div(maxP, 256)));
    pl.S_p = std::max(1, std::min(sp, kMaxPrefixSplits));
  }
  const int maxL = a->max_pages_per_branch * hpd::kPage;
  pl.S_s = std::max(1, std::min(ceil_div(maxL, kSuffixSplitKeys), kMaxSuffixSplits));
  const int rows_s = a->m * pl.G;
  pl.wr_s = rows_s <= 16 ? 1 : (rows_s <= 32 ? 2 : 4);
  pl.rt_s = ceil_div(rows_s, 16 * pl.wr_s);
  const size_t S = static_cast<size_t>(pl.S_p + pl.S_s);
  const size_t pairs = static_cast<size_t>(pl.rows_total) * a->H_q;
  pl.off_err = 0;
  pl.off_ctr = kAlign;
  pl.off_opart = align_up(pl.off_ctr + static_cast<size_t>(a->B) * a->H_kv * pl.rt_s * sizeof(int));
  pl.off_lpart = align_up(pl.off_opart + S * pairs * a->D * sizeof(float));
  pl.off_order = align_up(pl.off_lpart + S * pairs * sizeof(float));
  const size_t n_units =
      pl.use_tc ? static_cast<size_t>(std::max(pl.tiles_max, 0)) * a->H_kv * pl.S_p : 0;
  pl.bytes = align_up(pl.off_order + n_units * sizeof(int));
  return pl;
}

hpd_status check_accept_args(const void *logits, const int32_t *drafts, int B, int m, int V,
                             const int32_t *out_tokens, const int32_t *accepted_len) {
  if (!logits || !drafts || !out_tokens || !accepted_len) return HPD_ERR_INVALID_ARG;
  if (B < 1 || m < 1 || V < 1) return HPD_ERR_INVALID_ARG;
  if (m > 64) return HPD_ERR_UNSUPPORTED;
  if (!aligned(logits, 2) || !aligned(drafts, 4) || !aligned(out_tokens, 4) ||
      !aligned(accepted_len, 4))
    return HPD_ERR_INVALID_ARG;
  return HPD_OK;
}

// SM count of the current device (cached per device); 0 when unavailable.
int device_sms(int *dev_out) {
  static int sms[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  if (sms[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    sms[dev] = n;
  }
  if (dev_out) *dev_out = dev;
  return sms[dev];
}

// The attention kernel leaves SMs idle for part of its run: with fewer
// than two work units per SM its persistent CTAs (one per SM) either do not
// fill the GPU or finish their last round of whole units at different times.
// The acceptance then runs beside it on the idle SMs.  With more units per
// SM the dynamic scheduler keeps every SM busy until near the end and the
// two run in order.
constexpr int kConcurrentUnitsPerSm = 2;
bool step_concurrent(const hpd::Plan &pl, const hpd_branch_attn_args *a, int sms) {
  if (!pl.use_tc || sms <= 0) return false;
  const long long units = static_cast<long long>(pl.tiles_max) * a->H_kv * pl.S_p;
  return units < static_cast<long long>(kConcurrentUnitsPerSm) * sms;
}

// Per device: the second stream of hpd_decode_step and its fork / join
// events, created on the first call outside stream capture.
struct StepStreams {
  std::mutex mu;
  bool ready = false;
  cudaStream_t side = nullptr;
  cudaEvent_t fork = nullptr, join = nullptr;
};
StepStreams g_step[64];

}  // namespace

hpd_status hpd::record_cuda_error(cudaError_t e) { return cuda_fail(e); }

hpd_status hpd::check_call_args(const hpd_branch_attn_args *a) {
  const hpd_status st = check_scalars(a);
  if (st != HPD_OK) return st;
  if (!a->q || !a->prefix_cu || !a->branch_cu || !a->k_cache || !a->v_cache || !a->page_table ||
      !a->branch_len || !a->out)
    return HPD_ERR_INVALID_ARG;
  if (a->prefix_tokens > 0 && !a->prefix_page_table && (!a->prefix_k || !a->prefix_v))
    return HPD_ERR_INVALID_ARG;
  if (!aligned(a->q, 16) || !aligned(a->prefix_k, 16) || !aligned(a->prefix_v, 16) ||
      !aligned(a->k_cache, 16) || !aligned(a->v_cache, 16) || !aligned(a->out, 16) ||
      !aligned(a->lse, 4) || !aligned(a->prefix_cu, 4) || !aligned(a->branch_cu, 4) ||
      !aligned(a->page_table, 4) || !aligned(a->branch_len, 4) ||
      !aligned(a->branch_prefix_len, 4) || !aligned(a->prefix_page_table, 4))
    return HPD_ERR_INVALID_ARG;
  return HPD_OK;
}

size_t hpd::workspace_zero_bytes(const hpd_branch_attn_args *a) {
  if (check_scalars(a) != HPD_OK) return 0;
  return make_plan(a).off_opart;
}

extern "C" {

size_t hpd_branch_attn_workspace_size(const hpd_branch_attn_args *args) {
  if (check_scalars(args) != HPD_OK) return 0;
  return make_plan(args).bytes;
}

hpd_status hpd_workspace_init(void *workspace, size_t workspace_bytes, hpd_stream_t stream) {
  if (!workspace || !aligned(workspace, kAlign) || workspace_bytes < kAlign)
    return HPD_ERR_WORKSPACE;
  const cudaError_t e =
      cudaMemsetAsync(workspace, 0, workspace_bytes, reinterpret_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? HPD_OK : cuda_fail(e);
}

int hpd_branch_attn_launches(const hpd_branch_attn_args *args) {
  if (check_scalars(args) != HPD_OK) return 0;
  const hpd::Plan pl = make_plan(args);
  return pl.use_tc ? 1 + (pl.lpt ? 1 : 0) + (pl.S_p > 1 ? 1 : 0) : 2;
}

const char *hpd_branch_attn_kernel_name(const hpd_branch_attn_args *args, int k) {
  if (check_scalars(args) != HPD_OK) return nullptr;
  const hpd::Plan pl = make_plan(args);
  static const char *mma_names[] = {"prefix_stage", "suffix_merge"};
  if (!pl.use_tc) return k >= 0 && k < 2 ? mma_names[k] : nullptr;
  const char *tc_names[3];
  int n = 0;
  if (pl.lpt) tc_names[n++] = "unit_order";
  tc_names[n++] = "branch_attn_tc";
  if (pl.S_p > 1) tc_names[n++] = "merge_splits";
  return k >= 0 && k < n ? tc_names[k] : nullptr;
}

hpd_status hpd_branch_attn(const hpd_branch_attn_args *a, hpd_stream_t stream) {
  return hpd_branch_attn_marked(a, stream, nullptr);
}

hpd_status hpd_branch_attn_marked(const hpd_branch_attn_args *a, hpd_stream_t stream,
                                  void *const *ev) {
  const hpd_status st = hpd::check_call_args(a);
  if (st != HPD_OK) return st;
  const hpd::Plan pl = make_plan(a);
  if (!a->workspace || !aligned(a->workspace, kAlign) || a->workspace_bytes < pl.bytes)
    return HPD_ERR_WORKSPACE;

  uint8_t *ws = static_cast<uint8_t *>(a->workspace);
  hpd::AttnParams p{};
  p.q = static_cast<const __nv_bfloat16 *>(a->q);
  p.prefix_k = static_cast<const __nv_bfloat16 *>(a->prefix_k ? a->prefix_k : a->k_cache);
  p.prefix_v = static_cast<const __nv_bfloat16 *>(a->prefix_v ? a->prefix_v : a->v_cache);
  p.prefix_cu = a->prefix_cu;
  p.branch_cu = a->branch_cu;
  p.branch_prefix_len = a->branch_prefix_len;
  p.prefix_page_table = a->prefix_page_table;
  p.max_prefix_pages = a->prefix_page_table ? a->max_prefix_pages : 0;
  p.k_cache = static_cast<const __nv_bfloat16 *>(a->k_cache);
  p.v_cache = static_cast<const __nv_bfloat16 *>(a->v_cache);
  p.page_table = a->page_table;
  p.branch_len = a->branch_len;
  p.n_docs = a->n_docs;
  p.B = a->B;
  p.m = a->m;
  p.H_q = a->H_q;
  p.H_kv = a->H_kv;
  p.G = pl.G;
  p.D = a->D;
  p.num_pages = a->num_pages;
  p.max_pages = a->max_pages_per_branch;
  p.prefix_tokens = a->prefix_tokens;
  const float scale = a->scale != 0.f ? a->scale : 1.0f / std::sqrt(static_cast<float>(a->D));
  p.scale_log2 = scale * hpd::kLog2e;
  p.S_p = pl.S_p;
  p.S_s = pl.S_s;
  p.rows_total = pl.rows_total;
  p.o_part = reinterpret_cast<float *>(ws + pl.off_opart);
  p.l_part = reinterpret_cast<float *>(ws + pl.off_lpart);
  p.err = reinterpret_cast<uint32_t *>(ws + pl.off_err);
  p.counters = reinterpret_cast<int *>(ws + pl.off_ctr);
  p.unit_ctr = reinterpret_cast<int *>(ws + pl.off_err + 8);  // header: err word, then counters
  p.n_units = pl.tiles_max * a->H_kv * pl.S_p;
  p.unit_order = pl.lpt ? reinterpret_cast<int *>(ws + pl.off_order) : nullptr;
  p.out = static_cast<__nv_bfloat16 *>(a->out);
  p.out_align32 = aligned(a->out, 32);
  p.lse = a->lse;

  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // inside stream capture an event record becomes an external event node;
  // outside it, a plain record
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (ev) {
    const cudaError_t ce = cudaStreamIsCapturing(s, &cap);
    if (ce != cudaSuccess) return hpd::record_cuda_error(ce);
  }
  auto mark = [&](int k) -> cudaError_t {
    if (!ev || !ev[k]) return cudaSuccess;
    cudaEvent_t evk = static_cast<cudaEvent_t>(ev[k]);
    return cap == cudaStreamCaptureStatusActive
               ? cudaEventRecordWithFlags(evk, s, cudaEventRecordExternal)
               : cudaEventRecord(evk, s);
  };
  cudaError_t e = mark(0);
  if (pl.use_tc) {
    int k = 1;
    if (pl.lpt) {
      if (e == cudaSuccess)
        e = hpd::launch_unit_order(p, pl.tiles_max, const_cast<int *>(p.unit_order), s);
      if (e == cudaSuccess) e = mark(k++);
    }
    // each kernel after the first overlaps its launch with its predecessor
    if (e == cudaSuccess) e = hpd::launch_branch_attn_tc(p, pl, pl.lpt, s);
    if (e == cudaSuccess) e = mark(k++);
    if (pl.S_p > 1) {
      if (e == cudaSuccess) e = hpd::launch_merge_splits(p, true, s);
      if (e == cudaSuccess) e = mark(k++);
    }
  } else {
    if (e == cudaSuccess) e = hpd::launch_prefix_stage(p, pl, s);
    if (e == cudaSuccess) e = mark(1);
    if (e == cudaSuccess) e = hpd::launch_suffix_stage(p, pl, s);
    if (e == cudaSuccess) e = mark(2);
  }
  if (e != cudaSuccess) return cuda_fail(e);
  return HPD_OK;
}

hpd_status hpd_pmtp_accept(const void *logits, const int32_t *drafts, int B, int m, int V,
                           int32_t *out_tokens, int32_t *accepted_len, hpd_stream_t stream) {
  const hpd_status st = check_accept_args(logits, drafts, B, m, V, out_tokens, accepted_len);
  if (st != HPD_OK) return st;
  const cudaError_t e =
      hpd::launch_accept(static_cast<const __nv_bfloat16 *>(logits), drafts, B, m, V, out_tokens,
                         accepted_len, reinterpret_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? HPD_OK : cuda_fail(e);
}

int hpd_decode_step_concurrent(const hpd_branch_attn_args *args) {
  if (check_scalars(args) != HPD_OK) return -1;
  const int sms = device_sms(nullptr);
  if (sms <= 0) return -1;
  return step_concurrent(make_plan(args), args, sms) ? 1 : 0;
}

hpd_status hpd_decode_step(const hpd_branch_attn_args *a, const void *logits,
                           const int32_t *drafts, int V, int32_t *out_tokens,
                           int32_t *accepted_len, hpd_stream_t stream) {
  hpd_status st = hpd::check_call_args(a);
  if (st != HPD_OK) return st;
  st = check_accept_args(logits, drafts, a->B, a->m, V, out_tokens, accepted_len);
  if (st != HPD_OK) return st;
  const hpd::Plan pl = make_plan(a);
  if (!a->workspace || !aligned(a->workspace, kAlign) || a->workspace_bytes < pl.bytes)
    return HPD_ERR_WORKSPACE;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  auto accept_on = [&](cudaStream_t t) {
    return hpd::launch_accept(static_cast<const __nv_bfloat16 *>(logits), drafts, a->B, a->m, V,
                              out_tokens, accepted_len, t);
  };
  int dev = 0;
  const int sms = device_sms(&dev);
  if (!step_concurrent(pl, a, sms)) {
    st = hpd_branch_attn(a, stream);
    if (st != HPD_OK) return st;
    const cudaError_t e = accept_on(s);
    return e == cudaSuccess ? HPD_OK : cuda_fail(e);
  }
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  cudaError_t e = cudaStreamIsCapturing(s, &cap);
  if (e != cudaSuccess) return cuda_fail(e);
  StepStreams &ss = g_step[dev];
  std::lock_guard<std::mutex> lock(ss.mu);
  if (!ss.ready && cap == cudaStreamCaptureStatusNone) {
    e = cudaStreamCreateWithFlags(&ss.side, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ss.fork, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ss.join, cudaEventDisableTiming);
    if (e != cudaSuccess) return cuda_fail(e);
    ss.ready = true;
  }
  if (!ss.ready) {  // first call inside a capture: in order
    st = hpd_branch_attn(a, stream);
    if (st != HPD_OK) return st;
    e = accept_on(s);
    return e == cudaSuccess ? HPD_OK : cuda_fail(e);
  }
  // fork: the second stream waits for everything enqueued on `stream` so
  // far; the attention is enqueued first, then the acceptance beside it
  e = cudaEventRecord(ss.fork, s);
  if (e != cudaSuccess) return cuda_fail(e);
  e = cudaStreamWaitEvent(ss.side, ss.fork, 0);
  if (e != cudaSuccess) return cuda_fail(e);
  st = hpd_branch_attn(a, stream);
  cudaError_t ea = st == HPD_OK ? accept_on(ss.side) : cudaSuccess;
  // join (also after a failed launch, so that a capture is never left forked)
  e = cudaEventRecord(ss.join, ss.side);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(s, ss.join, 0);
  if (st != HPD_OK) return st;
  if (ea != cudaSuccess) return cuda_fail(ea);
  return e == cudaSuccess ? HPD_OK : cuda_fail(e);
}

hpd_status hpd_read_errors(const void *workspace, uint32_t *flags, hpd_stream_t stream) {
  if (!workspace || !flags || !aligned(workspace, kAlign)) return HPD_ERR_INVALID_ARG;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = cudaMemcpyAsync(flags, workspace, sizeof(uint32_t), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  return e == cudaSuccess ? HPD_OK : cuda_fail(e);
}

hpd_status hpd_wait_selftest(void *workspace, uint32_t limit_us, hpd_stream_t stream) {
  if (!workspace || !aligned(workspace, kAlign) || limit_us < 1 || limit_us > 10000000u)
    return HPD_ERR_INVALID_ARG;
  const cudaError_t e = hpd::launch_wait_selftest(static_cast<uint32_t *>(workspace),
                                                  static_cast<uint64_t>(limit_us) * 1000u,
                                                  reinterpret_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? HPD_OK : cuda_fail(e);
}

const char *hpd_status_string(hpd_status status) {
  switch (status) {
    case HPD_OK: return "ok";
    case HPD_ERR_INVALID_ARG: return "invalid argument";
    case HPD_ERR_UNSUPPORTED: return "unsupported shape";
    case HPD_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    case HPD_ERR_CUDA: return "CUDA error";
    case HPD_ERR_TIMEOUT: return "device-side wait timed out";
  }
  return "unknown status";
}

int hpd_last_cuda_error(void) { return g_last_cuda_error; }

int hpd_version(void) { return 100; }

}  // extern "C"
