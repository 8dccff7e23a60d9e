// prefix_tc.cu -- the shared-prefix stage on 5th-generation tensor cores.
//
// What it computes is the shared-prefix part of each branch's attention
// (Sec. 3.3): all query rows of a page's branches that read KV head g are
// stacked (row r <-> token branch_cu[d]*m + r/G, query head g*G + r%G) and
// attend to the page's prefix keys [0, P_d) -- masked per row at the
// branch's fork-position prefix length -- producing, per key chunk, the
// normalised partial output O_s (fp32) and lse_s (natural log) that the LSE
// merge combines with the private-suffix partials.
//
// How: one CTA owns 128 stacked rows x one key chunk of one (page, KV head).
//   warp 0      TMA producer: Q once, then 128-key K and V tiles into a
//               two-stage ring (128-byte swizzled, one box per 64 columns)
//   warp 1      TMEM owner and MMA issuer (one thread):
//                 S_j = Q K_j^T  -> TMEM, double buffered (2 x 128 columns)
//                 O  += P_j V_j  with P_j read from TMEM (bf16, written over
//                                S_j) and O accumulated in TMEM
//   warps 2-5   softmax: thread t of warp w owns TMEM lane 32*(w%4)+t, i.e.
//               one query row, so row max / sum need no shuffles.  O is
//               rescaled in TMEM only when a row's running max grows by more
//               than 2^8 (the stale max stays exact after the final
//               normalisation).
// All waits are bounded; a timeout sets HPD_DEVERR_TIMEOUT and the CTA
// drains its in-flight copies and MMAs, frees its TMEM and exits.
#include <cudaTypedefs.h>

#include <atomic>
#include <mutex>

#include "common.cuh"
#include "sm100.cuh"

namespace hpd {
namespace {

using namespace sm100;

constexpr int kRows = 128;        // stacked query rows per CTA (MMA M)
constexpr int kBlk = 128;         // keys per block (MMA N of S = Q K^T)
constexpr int kThreadsTc = 192;   // 6 warps
constexpr uint32_t kTmemCols = 512;
// TMEM columns: S / P double buffer at col_s(0) = 0 and col_s(1) = 128, O at 256.
__host__ __device__ constexpr uint32_t col_s(int s) { return s ? 128u : 0u; }
constexpr uint32_t kColO = 256;
constexpr float kRescaleLog2 = 8.0f;  // tolerate a stale row max up to 2^8

template <int D>
struct TcLayout {
  static constexpr int kChunks = D / 64;                   // 64-column (128-byte) boxes
  static constexpr uint32_t kChunkBytes = kRows * 128;     // 128 rows x 128 bytes
  static constexpr uint32_t kTileBytes = kChunks * kChunkBytes;
  static constexpr uint32_t kQ = 0;
  static constexpr uint32_t kK = kTileBytes;               // 2 stages
  static constexpr uint32_t kV = kK + 2 * kTileBytes;      // 2 stages
  static constexpr uint32_t kBytes = kV + 2 * kTileBytes;
  static constexpr uint32_t kDynSmem = kBytes + 1024;      // slack to align to 1024
};

struct __align__(8) TcShared {
  uint64_t q_full;
  uint64_t k_full[2];
  uint64_t v_full[2];
  uint64_t kv_empty[2];
  uint64_t s_full[2];
  uint64_t p_full[2];
  uint64_t pv_done;
  uint64_t mma_done;
  uint32_t tmem_base;
  int abort;
  int info[4];
  int kmax;
};

__device__ __forceinline__ void set_abort(TcShared &sh, uint32_t *err) {
  atomicExch(&sh.abort, 1);
  flag_error(err, HPD_DEVERR_TIMEOUT);
}

template <int D>
__global__ void __launch_bounds__(kThreadsTc, 1)
    prefix_tc_kernel(const __grid_constant__ CUtensorMap tm_q,
                     const __grid_constant__ CUtensorMap tm_k,
                     const __grid_constant__ CUtensorMap tm_v, const AttnParams p) {
  using L = TcLayout<D>;
  extern __shared__ uint8_t smem_raw[];
  __shared__ TcShared sh;
  const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = p.G, m = p.m;
  const int TT = kRows / G;  // tokens per row tile
  const float NEG_INF = -__int_as_float(0x7f800000);
  const int g = blockIdx.y, split = blockIdx.z, tile = blockIdx.x;

  // ------------------------------------------------------ work decode --
  if (tid == 0) {
    sh.info[0] = -1;
    sh.abort = 0;
  }
  __syncthreads();
  if (warp == 0) {
    // page owning this tile: page d has ceil(#branches(d) * m / TT) tiles
    int base = 0;
    for (int d0 = 0; d0 < p.n_docs; d0 += 32) {
      const int d = d0 + lane;
      int tiles = 0, b0 = 0, b1 = 0;
      if (d < p.n_docs) {
        b0 = min(max(p.branch_cu[d], 0), p.B);
        b1 = min(max(p.branch_cu[d + 1], 0), p.B);
        if (b1 < b0) {
          flag_error(p.err, HPD_DEVERR_BRANCH_CU);
          b1 = b0;
        }
        tiles = ceil_div_i((b1 - b0) * m, TT);
      }
      int incl = tiles;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += v;
      }
      const int excl = incl - tiles;
      if (tiles > 0 && tile >= base + excl && tile < base + incl) {
        sh.info[0] = d;
        sh.info[1] = tile - base - excl;
        sh.info[2] = b0;
        sh.info[3] = b1;
      }
      base += __shfl_sync(0xffffffffu, incl, 31);
      if (base > tile) break;
    }
  }
  __syncthreads();
  const int d = sh.info[0];
  if (d < 0) return;
  const int lt = sh.info[1], b0 = sh.info[2], b1 = sh.info[3];
  const int a0 = p.prefix_cu[d], a1 = p.prefix_cu[d + 1];
  if (tid == 0 && (a0 < 0 || a1 < a0 || a1 > p.prefix_tokens))
    flag_error(p.err, HPD_DEVERR_PREFIX_CU);
  const int pc0 = min(max(a0, 0), p.prefix_tokens);
  const int pc1 = min(max(a1, pc0), p.prefix_tokens);
  const int P_d = pc1 - pc0;
  const int tok0 = b0 * m + lt * TT;
  const int ntok = min(TT, (b1 - b0) * m - lt * TT);
  const int nrows = ntok * G;
  const int chunk = ceil_div_i(ceil_div_i(max(P_d, 1), p.S_p), kBlk) * kBlk;
  const int k_begin = split * chunk;
  int k_end = min(P_d, k_begin + chunk);

  auto out_index = [&](int r) -> size_t {
    const int token = tok0 + r / G;
    const int head = g * G + r % G;
    return (static_cast<size_t>(split) * p.rows_total + token) * p.H_q + head;
  };
  // exclusive key limit of stacked row r (fork-position prefix, chunk end)
  auto row_limit = [&](int r) -> int {
    if (r >= nrows) return k_begin;
    int lim = k_end;
    if (p.branch_prefix_len) {
      const int b = (tok0 + r / G) / m;
      int f = p.branch_prefix_len[b];
      if (f < 0 || f > P_d) {
        flag_error(p.err, HPD_DEVERR_FORK_LEN);
        f = min(max(f, 0), P_d);
      }
      lim = min(lim, f);
    }
    return lim;
  };
  if (p.branch_prefix_len) {
    if (tid == 0) sh.kmax = k_begin;
    __syncthreads();
    if (tid < kRows) atomicMax(&sh.kmax, row_limit(tid));
    __syncthreads();
    k_end = min(k_end, sh.kmax);
  }
  if (nrows <= 0) return;
  if (k_end <= k_begin) {
    for (int r = tid; r < nrows; r += kThreadsTc) p.l_part[out_index(r)] = NEG_INF;
    return;
  }
  const int n_blocks = ceil_div_i(k_end - k_begin, kBlk);

  // ------------------------------------------------------------- setup --
  const uint32_t b_q = smem_u32(&sh.q_full);
  auto bar = [](uint64_t &b) { return smem_u32(&b); };
  if (tid == 0) {
    mbar_init(b_q, 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(bar(sh.k_full[s]), 1);
      mbar_init(bar(sh.v_full[s]), 1);
      mbar_init(bar(sh.kv_empty[s]), 1);
      mbar_init(bar(sh.s_full[s]), 1);
      mbar_init(bar(sh.p_full[s]), 4);  // one arrival per softmax warp
    }
    mbar_init(bar(sh.pv_done), 1);
    mbar_init(bar(sh.mma_done), 1);
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&sh.tmem_base), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sh.tmem_base;

  if (warp == 0) {
    // ------------------------------------------------------ producer --
    if (lane == 0) {
      prefetch_tmap(&tm_q);
      prefetch_tmap(&tm_k);
      prefetch_tmap(&tm_v);
      mbar_arrive_expect_tx(b_q, L::kTileBytes);
      for (int c = 0; c < L::kChunks; ++c)
        tma_load_3d(sbase + L::kQ + c * L::kChunkBytes, &tm_q, b_q, c * 64, g * G, tok0);
      int issued = 0;
      for (int j = 0; j < n_blocks; ++j) {
        const int s = j & 1;
        if (j >= 2) {
          if (sh.abort || !mbar_wait(bar(sh.kv_empty[s]), ((j >> 1) - 1) & 1)) {
            set_abort(sh, p.err);
            break;
          }
        }
        const int key = pc0 + k_begin + j * kBlk;
        mbar_arrive_expect_tx(bar(sh.k_full[s]), L::kTileBytes);
        for (int c = 0; c < L::kChunks; ++c)
          tma_load_3d(sbase + L::kK + s * L::kTileBytes + c * L::kChunkBytes, &tm_k,
                      bar(sh.k_full[s]), c * 64, g, key);
        mbar_arrive_expect_tx(bar(sh.v_full[s]), L::kTileBytes);
        for (int c = 0; c < L::kChunks; ++c)
          tma_load_3d(sbase + L::kV + s * L::kTileBytes + c * L::kChunkBytes, &tm_v,
                      bar(sh.v_full[s]), c * 64, g, key);
        issued = j + 1;
      }
      // Do not leave while a copy into this CTA's shared memory is in flight.
      mbar_wait(b_q, 0);
      for (int j = max(0, issued - 2); j < issued; ++j) {
        mbar_wait(bar(sh.k_full[j & 1]), (j >> 1) & 1);
        mbar_wait(bar(sh.v_full[j & 1]), (j >> 1) & 1);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------- MMA issuer --
    if (lane == 0) {
      constexpr uint32_t idesc_qk = idesc_bf16_f32(kRows, kBlk, false);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(kRows, 64, true);
      bool ok = mbar_wait(b_q, 0);
      tc_fence_after();
      for (int j = 0; ok && j <= n_blocks; ++j) {
        if (j < n_blocks) {
          const int s = j & 1;
          if (sh.abort || !mbar_wait(bar(sh.k_full[s]), (j >> 1) & 1)) { ok = false; break; }
          tc_fence_after();
          const uint32_t kb = sbase + L::kK + s * L::kTileBytes;
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t off = (kk >> 2) * L::kChunkBytes + (kk & 3) * 32;
            mma_ss(tmem + col_s(s), smem_desc_sw128(sbase + L::kQ + off, 16, 1024),
                   smem_desc_sw128(kb + off, 16, 1024), idesc_qk, kk > 0);
          }
          mma_commit(bar(sh.s_full[s]));
        }
        if (j >= 1) {
          const int jj = j - 1, s = jj & 1;
          if (sh.abort || !mbar_wait(bar(sh.p_full[s]), (jj >> 1) & 1) ||
              !mbar_wait(bar(sh.v_full[s]), (jj >> 1) & 1)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t vb = sbase + L::kV + s * L::kTileBytes;
          // One N = 64 MMA per 64-column V box: each reads a single 128-byte
          // swizzle atom along N (MN-major B), 8-key groups 1024 bytes apart.
#pragma unroll
          for (int kk = 0; kk < kBlk / 16; ++kk) {
#pragma unroll
            for (int c = 0; c < L::kChunks; ++c) {
              mma_ts(tmem + kColO + c * 64, tmem + col_s(s) + kk * 8,
                     smem_desc_sw128(vb + c * L::kChunkBytes + kk * 16 * 128, 16, 1024),
                     idesc_pv, (jj > 0 || kk > 0) ? 1u : 0u);
            }
          }
          mma_commit(bar(sh.kv_empty[s]));
          mma_commit(bar(sh.pv_done));
        }
      }
      if (!ok) set_abort(sh, p.err);
      // every MMA issued above has finished before TMEM is released
      mma_commit(bar(sh.mma_done));
      mbar_wait(bar(sh.mma_done), 0);
    }
  } else {
    // ------------------------------------------------------- softmax --
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    const uint32_t t_lane = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    const int lim = row_limit(row);
    const float sl2 = p.scale_log2;
    float m_run = NEG_INF, l_run = 0.f;
    bool ok = true;
    for (int j = 0; j < n_blocks; ++j) {
      const int s = j & 1;
      if (sh.abort || !mbar_wait(bar(sh.s_full[s]), (j >> 1) & 1)) { ok = false; break; }
      tc_fence_after();
      uint32_t v[kBlk];
#pragma unroll
      for (int c = 0; c < kBlk; c += 32) tmem_ld32(t_lane + col_s(s) + c, v + c);
      tmem_ld_wait();
      const int key0 = k_begin + j * kBlk;
      float mx = NEG_INF;
      if (key0 + kBlk <= lim) {
#pragma unroll
        for (int c = 0; c < kBlk; ++c) {
          const float f = __uint_as_float(v[c]) * sl2;
          v[c] = __float_as_uint(f);
          mx = fmaxf(mx, f);
        }
      } else {
#pragma unroll
        for (int c = 0; c < kBlk; ++c) {
          const float f = key0 + c < lim ? __uint_as_float(v[c]) * sl2 : NEG_INF;
          v[c] = __float_as_uint(f);
          mx = fmaxf(mx, f);
        }
      }
      const float m_new = mx > m_run + kRescaleLog2 ? mx : m_run;
      const float base = m_new == NEG_INF ? 0.f : m_new;
      const float alpha = m_new == m_run ? 1.f : fast_exp2(m_run - base);
      float sum = 0.f;
      uint32_t pk[kBlk / 2];
#pragma unroll
      for (int c = 0; c < kBlk; c += 2) {
        const float e0 = fast_exp2(__uint_as_float(v[c]) - base);
        const float e1 = fast_exp2(__uint_as_float(v[c + 1]) - base);
        sum += e0 + e1;
        pk[c / 2] = pack_bf16x2(e0, e1);
      }
      l_run = l_run * alpha + sum;
      m_run = m_new;
      tmem_st32(t_lane + col_s(s), pk);
      tmem_st32(t_lane + col_s(s) + 32, pk + 32);
      // pv_done completes once per PV_j; waiting on every phase in order
      // keeps this warp at most one phase behind, so parity waits are exact.
      if (j > 0 && !mbar_wait(bar(sh.pv_done), (j - 1) & 1)) { ok = false; break; }
      // Rescale O (PV_{j-1} has landed) if any row of this warp needs it.
      if (__any_sync(0xffffffffu, j > 0 && alpha != 1.f)) {
        tc_fence_after();
#pragma unroll
        for (int c = 0; c < D; c += 32) {
          uint32_t o[32];
          tmem_ld32(t_lane + kColO + c, o);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
          tmem_st32(t_lane + kColO + c, o);
        }
      }
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(sh.p_full[s]));
    }
    if (!ok) set_abort(sh, p.err);
    // ---------------------------------------------------- epilogue --
    if (ok && mbar_wait(bar(sh.pv_done), (n_blocks - 1) & 1)) {
      tc_fence_after();
      const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
      float *dst = row < nrows ? p.o_part + out_index(row) * D : nullptr;
#pragma unroll
      for (int c = 0; c < D; c += 32) {
        uint32_t o[32];
        tmem_ld32(t_lane + kColO + c, o);
        tmem_ld_wait();
        if (dst) {
#pragma unroll
          for (int e = 0; e < 32; e += 4)
            *reinterpret_cast<float4 *>(dst + c + e) =
                make_float4(__uint_as_float(o[e]) * inv, __uint_as_float(o[e + 1]) * inv,
                            __uint_as_float(o[e + 2]) * inv, __uint_as_float(o[e + 3]) * inv);
        }
      }
      if (dst) p.l_part[out_index(row)] = l_run > 0.f ? (m_run + __log2f(l_run)) * kLn2 : NEG_INF;
    } else if (ok) {
      set_abort(sh, p.err);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ------------------------------------------------------------------ host --
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
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

// 3-D bf16 tensor map [d2][d1][d0] (d0 contiguous), 128-byte swizzle.
cudaError_t make_map(CUtensorMap *map, const void *base, uint64_t d0, uint64_t d1, uint64_t d2,
                     uint32_t b0, uint32_t b1, uint32_t b2) {
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

template <int D>
cudaError_t launch_tc(const AttnParams &p, const Plan &plan, cudaStream_t s) {
  using L = TcLayout<D>;
  CUtensorMap tq, tk, tv;
  const int G = p.G;
  cudaError_t e = make_map(&tq, p.q, D, p.H_q, static_cast<uint64_t>(p.rows_total), 64, G,
                           kRows / G);
  if (e != cudaSuccess) return e;
  const bool has_prefix = p.prefix_tokens > 0;
  const uint64_t T = has_prefix ? static_cast<uint64_t>(p.prefix_tokens) : 1;
  e = make_map(&tk, has_prefix ? p.prefix_k : p.k_cache, D, p.H_kv, T, 64, 1, kBlk);
  if (e != cudaSuccess) return e;
  e = make_map(&tv, has_prefix ? p.prefix_v : p.v_cache, D, p.H_kv, T, 64, 1, kBlk);
  if (e != cudaSuccess) return e;

  static std::atomic<uint64_t> configured{0};
  int dev = 0;
  e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(configured.load(std::memory_order_acquire) & bit)) {
    e = cudaFuncSetAttribute(prefix_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(L::kDynSmem));
    if (e != cudaSuccess) return e;
    configured.fetch_or(bit, std::memory_order_acq_rel);
  }
  const dim3 grid(plan.tiles_max, p.H_kv, plan.S_p);
  prefix_tc_kernel<D><<<grid, kThreadsTc, L::kDynSmem, s>>>(tq, tk, tv, p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_prefix_stage_tc(const AttnParams &p, const Plan &plan, cudaStream_t s) {
  if (plan.tiles_max <= 0) return cudaSuccess;
  return p.D == 64 ? launch_tc<64>(p, plan, s) : launch_tc<128>(p, plan, s);
}

}  // namespace hpd
