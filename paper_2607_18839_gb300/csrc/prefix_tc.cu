// prefix_tc.cu -- the shared-prefix stage on 5th-generation tensor cores.
//
// What it computes is the shared-prefix part of each branch's attention
// (Sec. 3.3): all query rows of a page's branches that read KV head g are
// stacked (row r <-> token branch_cu[d]*m + r/G, query head g*G + r%G) and
// attend to the page's prefix keys [0, P_d) -- masked per row at the
// branch's fork-position prefix length -- producing, per key split, the
// normalised partial output O_s (fp32) and lse_s (natural log) that the LSE
// merge combines with the private-suffix partials.
//
// How: one CTA owns NT tiles of 128 stacked rows (NT = 1 or 2) and one key
// split of one (page, KV head).  Each 128-key K / V tile is loaded once and
// used by all NT row tiles.
//   warp 0      TMA producer: the Q tiles once, then K and V tiles into
//               two-stage rings (128-byte swizzled, one box per 64 columns).
//               A K stage is refilled as soon as its Q K^T MMAs finish, a V
//               stage once its P V MMAs finish.
//   warp 1      TMEM owner and MMA issuer (one thread):
//                 S = Q K_j^T  -> TMEM (fp32, 128 columns per tile)
//                 O += P_j V_j  with P_j read from TMEM (bf16, written over
//                               S) and O accumulated in TMEM
//               NT = 1: S is double buffered, so Q K_{j+1}^T runs while the
//               softmax works on block j.  NT = 2: the two tiles alternate,
//               so one tile's MMAs run while the other tile's softmax works.
//   warps 2..   softmax, one warpgroup per tile: thread t of warp w owns TMEM
//               lane 32*(w%4)+t, i.e. one query row, so row max / sum need
//               no shuffles.  O is rescaled in TMEM only when a row's running
//               max grows by more than 2^8; the stale max stays exact after
//               the final normalisation.
// All waits are bounded; a timeout sets HPD_DEVERR_TIMEOUT and the CTA
// drains its in-flight copies and MMAs, frees its TMEM and exits.
#include <atomic>

#include "tc_common.cuh"

namespace hpd {
namespace {

using namespace sm100;
using tc::kBlk;
using tc::kRows;

constexpr uint32_t kTmemCols = 512;

template <int D, int NT>
struct TcLayout {
  static constexpr int kChunks = D / 64;                // 64-column (128-byte) boxes
  static constexpr uint32_t kChunkBytes = kRows * 128;  // 128 rows x 128 bytes
  static constexpr uint32_t kTileBytes = kChunks * kChunkBytes;
  static constexpr uint32_t kQ = 0;                     // NT tiles
  static constexpr uint32_t kK = NT * kTileBytes;       // 2 stages
  static constexpr uint32_t kV = kK + 2 * kTileBytes;   // 2 stages
  static constexpr uint32_t kBytes = kV + 2 * kTileBytes;
  static constexpr uint32_t kDynSmem = kBytes + 1024;   // slack to align to 1024
  static constexpr int kThreads = 32 * (2 + 4 * NT);
  // TMEM columns: S of buffer / tile i at col_s(i), O of tile t at col_o(t).
  static __device__ __forceinline__ uint32_t col_s(int i) { return i ? 128u : 0u; }
  static __device__ __forceinline__ uint32_t col_o(int t) { return t ? 384u : 256u; }
};

struct __align__(8) TcShared {
  uint64_t q_full;
  uint64_t k_full[2], v_full[2];
  uint64_t k_empty[2], v_empty[2];
  uint64_t s_full[2];   // NT = 1: per S buffer; NT = 2: per tile
  uint64_t p_full[2];   // same indexing as s_full
  uint64_t pv_done[2];  // per tile
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

template <int D, int NT>
__global__ void __launch_bounds__(TcLayout<D, NT>::kThreads, 1)
    prefix_tc_kernel(const __grid_constant__ CUtensorMap tm_q,
                     const __grid_constant__ CUtensorMap tm_k,
                     const __grid_constant__ CUtensorMap tm_v, const AttnParams p) {
  using L = TcLayout<D, NT>;
  extern __shared__ uint8_t smem_raw[];
  __shared__ TcShared sh;
  const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = p.G, m = p.m;
  const int TT = kRows / G;  // tokens per 128-row tile
  const float NEG_INF = -__int_as_float(0x7f800000);
  const int g = blockIdx.y, split = blockIdx.z;

  // ------------------------------------------------------ work decode --
  if (tid == 0) {
    sh.info[0] = -1;
    sh.abort = 0;
  }
  __syncthreads();
  if (warp == 0) tc::locate_tile(p, blockIdx.x, NT * TT, sh.info);
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
  const int tok0 = b0 * m + lt * NT * TT;
  const int ntok = min(NT * TT, (b1 - b0) * m - lt * NT * TT);
  const int nrows = ntok * G;
  const int n_act = NT == 1 ? 1 : (nrows > kRows ? 2 : 1);  // row tiles holding rows
  int k_begin, k_end;
  tc::split_range(P_d, p.S_p, split, k_begin, k_end);

  auto out_index = [&](int r) -> size_t {
    const int token = tok0 + r / G;
    const int head = g * G + r % G;
    return (static_cast<size_t>(split) * p.rows_total + token) * p.H_q + head;
  };
  // exclusive key limit of CTA row r (fork-position prefix, split end)
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
    for (int r = tid; r < NT * kRows; r += L::kThreads) atomicMax(&sh.kmax, row_limit(r));
    __syncthreads();
    k_end = min(k_end, sh.kmax);
  }
  if (nrows <= 0) return;
  if (k_end <= k_begin) {
    for (int r = tid; r < nrows; r += L::kThreads) p.l_part[out_index(r)] = NEG_INF;
    return;
  }
  const int n_blocks = ceil_div_i(k_end - k_begin, kBlk);

  // ------------------------------------------------------------- setup --
  auto bar = [](uint64_t &b) { return smem_u32(&b); };
  if (tid == 0) {
    mbar_init(bar(sh.q_full), 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(bar(sh.k_full[s]), 1);
      mbar_init(bar(sh.v_full[s]), 1);
      mbar_init(bar(sh.k_empty[s]), 1);
      mbar_init(bar(sh.v_empty[s]), 1);
      mbar_init(bar(sh.s_full[s]), 1);
      mbar_init(bar(sh.p_full[s]), 4);  // one arrival per softmax warp
      mbar_init(bar(sh.pv_done[s]), 1);
    }
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
      mbar_arrive_expect_tx(bar(sh.q_full), NT * L::kTileBytes);
      for (int t = 0; t < NT; ++t)
        for (int c = 0; c < L::kChunks; ++c)
          tma_load_3d(sbase + L::kQ + t * L::kTileBytes + c * L::kChunkBytes, &tm_q,
                      bar(sh.q_full), c * 64, g * G, tok0 + t * TT);
      int issued_k = 0, issued_v = 0;
      for (int j = 0; j < n_blocks; ++j) {
        const int s = j & 1, prev = ((j >> 1) - 1) & 1;
        const int key = pc0 + k_begin + j * kBlk;
        if (j >= 2 && (sh.abort || !mbar_wait(bar(sh.k_empty[s]), prev))) {
          set_abort(sh, p.err);
          break;
        }
        mbar_arrive_expect_tx(bar(sh.k_full[s]), L::kTileBytes);
        for (int c = 0; c < L::kChunks; ++c)
          tma_load_3d(sbase + L::kK + s * L::kTileBytes + c * L::kChunkBytes, &tm_k,
                      bar(sh.k_full[s]), c * 64, g, key);
        issued_k = j + 1;
        if (j >= 2 && (sh.abort || !mbar_wait(bar(sh.v_empty[s]), prev))) {
          set_abort(sh, p.err);
          break;
        }
        mbar_arrive_expect_tx(bar(sh.v_full[s]), L::kTileBytes);
        for (int c = 0; c < L::kChunks; ++c)
          tma_load_3d(sbase + L::kV + s * L::kTileBytes + c * L::kChunkBytes, &tm_v,
                      bar(sh.v_full[s]), c * 64, g, key);
        issued_v = j + 1;
      }
      // Do not leave while a copy into this CTA's shared memory is in flight.
      mbar_wait(bar(sh.q_full), 0);
      for (int j = max(0, issued_k - 2); j < issued_k; ++j)
        mbar_wait(bar(sh.k_full[j & 1]), (j >> 1) & 1);
      for (int j = max(0, issued_v - 2); j < issued_v; ++j)
        mbar_wait(bar(sh.v_full[j & 1]), (j >> 1) & 1);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------- MMA issuer --
    if (lane == 0) {
      constexpr uint32_t idesc_qk = idesc_bf16_f32(kRows, kBlk, false);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(kRows, 64, true);
      // S[col] = Q_t K_j^T
      auto issue_qk = [&](int t, int j, uint32_t col) {
        const uint32_t qb = sbase + L::kQ + t * L::kTileBytes;
        const uint32_t kb = sbase + L::kK + (j & 1) * L::kTileBytes;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (kk >> 2) * L::kChunkBytes + (kk & 3) * 32;
          mma_ss(tmem + col, smem_desc_sw128(qb + off, 16, 1024),
                 smem_desc_sw128(kb + off, 16, 1024), idesc_qk, kk > 0);
        }
      };
      // O_t += P V_j with P in TMEM at column pcol.  One N = 64 MMA per
      // 64-column V box: each reads a single 128-byte swizzle atom along N
      // (MN-major B), 8-key groups 1024 bytes apart.
      auto issue_pv = [&](int t, int j, uint32_t pcol) {
        const uint32_t vb = sbase + L::kV + (j & 1) * L::kTileBytes;
#pragma unroll
        for (int kk = 0; kk < kBlk / 16; ++kk) {
#pragma unroll
          for (int c = 0; c < L::kChunks; ++c)
            mma_ts(tmem + L::col_o(t) + c * 64, tmem + pcol + kk * 8,
                   smem_desc_sw128(vb + c * L::kChunkBytes + kk * 16 * 128, 16, 1024), idesc_pv,
                   (j > 0 || kk > 0) ? 1u : 0u);
        }
      };
      auto wait = [&](uint64_t &b, int parity) {
        if (sh.abort || !mbar_wait(bar(b), parity)) return false;
        tc_fence_after();
        return true;
      };
      bool ok = wait(sh.q_full, 0);
      if constexpr (NT == 1) {
        for (int j = 0; ok && j <= n_blocks; ++j) {
          if (j < n_blocks) {
            const int s = j & 1;
            if (!(ok = wait(sh.k_full[s], (j >> 1) & 1))) break;
            issue_qk(0, j, L::col_s(s));
            mma_commit(bar(sh.s_full[s]));
            mma_commit(bar(sh.k_empty[s]));
          }
          if (j >= 1) {
            const int jj = j - 1, s = jj & 1;
            if (!(ok = wait(sh.p_full[s], (jj >> 1) & 1) && wait(sh.v_full[s], (jj >> 1) & 1)))
              break;
            issue_pv(0, jj, L::col_s(s));
            mma_commit(bar(sh.pv_done[0]));
            mma_commit(bar(sh.v_empty[s]));
          }
        }
      } else {
        // tile t's S lives at col_s(t); tiles alternate on the tensor pipe:
        //   PV_0(j)  QK_0(j+1)  PV_1(j)  QK_1(j+1)  ...
        if (ok && (ok = wait(sh.k_full[0], 0))) {
          for (int t = 0; t < n_act; ++t) {
            issue_qk(t, 0, L::col_s(t));
            mma_commit(bar(sh.s_full[t]));
          }
          mma_commit(bar(sh.k_empty[0]));
        }
        for (int j = 0; ok && j < n_blocks; ++j) {
          const int s = j & 1;
          const bool more = j + 1 < n_blocks;
          for (int t = 0; t < n_act; ++t) {
            if (!(ok = wait(sh.p_full[t], j & 1))) break;
            if (t == 0 && !(ok = wait(sh.v_full[s], (j >> 1) & 1))) break;
            issue_pv(t, j, L::col_s(t));
            mma_commit(bar(sh.pv_done[t]));
            if (more) {
              if (t == 0 && !(ok = wait(sh.k_full[s ^ 1], ((j + 1) >> 1) & 1))) break;
              issue_qk(t, j + 1, L::col_s(t));
              mma_commit(bar(sh.s_full[t]));
            }
          }
          if (!ok) break;
          mma_commit(bar(sh.v_empty[s]));
          if (more) mma_commit(bar(sh.k_empty[s ^ 1]));
        }
      }
      if (!ok) set_abort(sh, p.err);
      // every MMA issued above has finished before TMEM is released
      mma_commit(bar(sh.mma_done));
      mbar_wait(bar(sh.mma_done), 0);
    }
  } else {
    // ------------------------------------------------------- softmax --
    const int t = (warp - 2) >> 2;  // row tile of this warpgroup
    const int quad = warp & 3;      // TMEM lane quadrant this warp may access
    const int row = t * kRows + quad * 32 + lane;
    const uint32_t t_lane = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    const uint32_t o_col = L::col_o(t);
    if (t < n_act) {
      const int lim = row_limit(row);
      const float sl2 = p.scale_log2;
      float m_run = NEG_INF, l_run = 0.f;
      bool ok = true;
      for (int j = 0; j < n_blocks; ++j) {
        const int si = NT == 1 ? (j & 1) : t;  // S buffer / barrier index
        const int ph = NT == 1 ? ((j >> 1) & 1) : (j & 1);
        const uint32_t s_col = L::col_s(si);
        if (sh.abort || !mbar_wait(bar(sh.s_full[si]), ph)) { ok = false; break; }
        tc_fence_after();
        uint32_t v[kBlk];
#pragma unroll
        for (int c = 0; c < kBlk; c += 32) tmem_ld32(t_lane + s_col + c, v + c);
        tmem_ld_wait();
        uint32_t pk[kBlk / 2];
        const float alpha = tc::softmax_block(v, k_begin + j * kBlk, lim, sl2, m_run, l_run, pk);
        tmem_st32(t_lane + s_col, pk);
        tmem_st32(t_lane + s_col + 32, pk + 32);
        // pv_done[t] completes once per block; waiting on every phase in
        // order keeps this warp at most one phase behind, so parity is exact.
        if (j > 0 && !mbar_wait(bar(sh.pv_done[t]), (j - 1) & 1)) { ok = false; break; }
        // Rescale O (PV of block j-1 has landed) if any row of this warp needs it.
        if (__any_sync(0xffffffffu, j > 0 && alpha != 1.f)) {
          tc_fence_after();
#pragma unroll
          for (int c = 0; c < D; c += 32) {
            uint32_t o[32];
            tmem_ld32(t_lane + o_col + c, o);
            tmem_ld_wait();
#pragma unroll
            for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
            tmem_st32(t_lane + o_col + c, o);
          }
        }
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(sh.p_full[si]));
      }
      if (!ok) set_abort(sh, p.err);
      // -------------------------------------------------- epilogue --
      if (ok && mbar_wait(bar(sh.pv_done[t]), (n_blocks - 1) & 1)) {
        tc_fence_after();
        const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
        float *dst = row < nrows ? p.o_part + out_index(row) * D : nullptr;
#pragma unroll
        for (int c = 0; c < D; c += 32) {
          uint32_t o[32];
          tmem_ld32(t_lane + o_col + c, o);
          tmem_ld_wait();
          if (dst) {
#pragma unroll
            for (int e = 0; e < 32; e += 4)
              *reinterpret_cast<float4 *>(dst + c + e) =
                  make_float4(__uint_as_float(o[e]) * inv, __uint_as_float(o[e + 1]) * inv,
                              __uint_as_float(o[e + 2]) * inv, __uint_as_float(o[e + 3]) * inv);
          }
        }
        if (dst)
          p.l_part[out_index(row)] = l_run > 0.f ? (m_run + __log2f(l_run)) * kLn2 : NEG_INF;
      } else if (ok) {
        set_abort(sh, p.err);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

template <int D, int NT>
cudaError_t launch_tc(const AttnParams &p, const Plan &plan, cudaStream_t s) {
  using L = TcLayout<D, NT>;
  CUtensorMap tq, tk, tv;
  cudaError_t e = tc::make_prefix_maps(p, &tq, &tk, &tv);
  if (e != cudaSuccess) return e;
  static std::atomic<uint64_t> configured{0};
  int dev = 0;
  e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(configured.load(std::memory_order_acquire) & bit)) {
    e = cudaFuncSetAttribute(prefix_tc_kernel<D, NT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(L::kDynSmem));
    if (e != cudaSuccess) return e;
    configured.fetch_or(bit, std::memory_order_acq_rel);
  }
  const dim3 grid(plan.tiles_max, p.H_kv, plan.S_p);
  prefix_tc_kernel<D, NT><<<grid, L::kThreads, L::kDynSmem, s>>>(tq, tk, tv, p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_prefix_stage_tc(const AttnParams &p, const Plan &plan, cudaStream_t s) {
  if (plan.tiles_max <= 0) return cudaSuccess;
  if (plan.tc_tiles == 2)
    return p.D == 64 ? launch_tc<64, 2>(p, plan, s) : launch_tc<128, 2>(p, plan, s);
  return p.D == 64 ? launch_tc<64, 1>(p, plan, s) : launch_tc<128, 1>(p, plan, s);
}

}  // namespace hpd
