// branch_attn_tc.cu -- the branch-attention step on 5th-generation tensor
// cores: shared prefix and private suffixes in one kernel.
//
// What it computes (Sec. 3.3, "Dynamic Branch Forking and Efficient Context
// Isolation"; Sec. 3.4 for the m P-MTP queries): all query rows of a page's
// branches that read KV head g are stacked (row r <-> token
// branch_cu[d]*m + r/G, query head g*G + r%G).  Each row attends to
//   - the page's shared prefix keys [0, P_b), P_b its branch's fork-position
//     prefix length (P_d when none is given), and
//   - its own branch's private keys j <= L_b - m + i (i = the row's query).
// The page's prefix is read once per 128 or 256 stacked rows instead of once
// per branch: that is the shared-prefix KV reuse the method relies on.
//
// Key blocks: a CTA walks 128-key blocks of two kinds,
//   prefix blocks  128 consecutive prefix keys (3-D TMA box per 64 columns),
//   suffix blocks  8 pages of 16 keys, packed from the private caches of the
//                  CTA's branches in branch order (4-D TMA box per page).
// For every row and block the visible columns form one interval [lo, hi):
// a prefix block's keys below the row's limit, or the row's own branch's
// pages up to its causal bound.  Rows of other branches see nothing of a
// suffix page, so its probabilities are zero for them.
//
// How: one CTA owns NT tiles of 128 stacked rows (NT = 1 or 2) and one split
// (an even share of the blocks) of one (page, KV head).
//   warp 0      TMA producer: the Q tiles once, then K and V blocks into
//               two-stage rings (128-byte swizzled).  A K stage is refilled
//               as soon as its Q K^T MMAs finish, a V stage once its P V MMAs
//               finish.
//   warp 1      TMEM owner and MMA issuer (one thread):
//                 S = Q K^T   -> TMEM (fp32, 128 columns per tile)
//                 O += P V    with P read from TMEM (bf16, written over S) and
//                             O accumulated in TMEM
//               NT = 1: S is double buffered, so the next Q K^T runs while the
//               softmax works.  NT = 2: the two tiles alternate, so one
//               tile's MMAs run while the other tile's softmax works.
//   warps 2..   softmax, one warpgroup per tile: thread t of warp w owns TMEM
//               lane 32*(w%4)+t, i.e. one query row, so row max / sum need
//               no shuffles.  O is rescaled in TMEM only when a row's running
//               max grows by more than 2^8; the stale max stays exact after
//               the final normalisation.
// One split: the CTA writes the final bf16 output and lse.  Several splits:
// it writes its normalised fp32 partial and lse for merge.cu.
// All waits are bounded; a timeout sets HPD_DEVERR_TIMEOUT and the CTA
// drains its in-flight copies and MMAs, frees its TMEM and exits.
#include <algorithm>
#include <atomic>

#include "tc_common.cuh"

namespace hpd {
namespace {

using namespace sm100;
using tc::kBlk;
using tc::kRows;

constexpr uint32_t kTmemCols = 512;
constexpr int kMaxCtaBranches = 258;  // branches touching 256 stacked rows, + 1
constexpr int kPageCap = 4096;        // suffix page ids kept in shared memory
constexpr int kPagesPerBlock = kBlk / kPage;

template <int D, int NT>
struct TcLayout {
  static constexpr int kChunks = D / 64;                // 64-column (128-byte) boxes
  static constexpr uint32_t kChunkBytes = kRows * 128;  // 128 rows x 128 bytes
  static constexpr uint32_t kTileBytes = kChunks * kChunkBytes;
  static constexpr uint32_t kQ = 0;                     // NT tiles
  static constexpr uint32_t kK = NT * kTileBytes;       // 2 stages
  static constexpr uint32_t kV = kK + 2 * kTileBytes;   // 2 stages
  static constexpr uint32_t kPages = kV + 2 * kTileBytes;  // int32 [kPageCap]
  static constexpr uint32_t kBytes = kPages + kPageCap * 4;
  static constexpr uint32_t kDynSmem = kBytes + 1024;   // slack to align to 1024
  // softmax warpgroups per row tile: one tile per CTA splits every row's key
  // columns over two warpgroups; two tiles keep one warpgroup each (registers)
  static constexpr int kHalves = NT == 1 ? 2 : 1;
  static constexpr int kThreads = 32 * (2 + 4 * kHalves * NT);  // producer, MMA, softmax
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
  int unit;
  // the two column halves of every row exchange their partial row max
  // (double buffered by block parity) and, at the end, their partial sums
  float xmax[2][2][kRows];  // [half][block parity][row] (one-tile CTAs)
  float xsum[2][kRows];     // [half][row]
  int page_start[kMaxCtaBranches + 1];  // packed page offset of each CTA branch
  int blen[kMaxCtaBranches];            // private length L_b (clamped)
};

__device__ __forceinline__ void set_abort(TcShared &sh, uint32_t *err) {
  atomicExch(&sh.abort, 1);
  flag_error(err, HPD_DEVERR_TIMEOUT);
}

template <int D, int NT>
__global__ void __launch_bounds__(TcLayout<D, NT>::kThreads, 1)
    branch_attn_tc_kernel(const __grid_constant__ CUtensorMap tm_q,
                          const __grid_constant__ CUtensorMap tm_k,
                          const __grid_constant__ CUtensorMap tm_v,
                          const __grid_constant__ CUtensorMap tm_kc,
                          const __grid_constant__ CUtensorMap tm_vc, const AttnParams p) {
  using L = TcLayout<D, NT>;
  extern __shared__ uint8_t smem_raw[];
  __shared__ TcShared sh;
  const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
  int *page_tab = reinterpret_cast<int *>(smem_raw + (sbase - smem_u32(smem_raw)) + L::kPages);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = p.G, m = p.m;
  const int TT = kRows / G;  // tokens per 128-row tile
  const float NEG_INF = -__int_as_float(0x7f800000);
  auto bar = [](uint64_t &b) { return smem_u32(&b); };

  // ------------------------------------------------------ once per CTA --
  if (tid == 0) {
    sh.abort = 0;
    mbar_init(bar(sh.q_full), 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(bar(sh.k_full[s]), 1);
      mbar_init(bar(sh.v_full[s]), 1);
      mbar_init(bar(sh.k_empty[s]), 1);
      mbar_init(bar(sh.v_empty[s]), 1);
      mbar_init(bar(sh.s_full[s]), 1);
      mbar_init(bar(sh.p_full[s]), 4 * L::kHalves);  // one arrival per softmax warp of the tile
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

  // Running counts of this CTA's work, identical in every thread; barrier
  // phases continue from one unit to the next through them.
  int jbase = 0;            // blocks processed (K / V stages; NT = 1: S buffers)
  int jt[2] = {0, 0};       // blocks processed by row tile t (NT = 2)
  int uidx = 0;             // units processed (Q loads)

  // ------------------------------------------- persistent loop over units --
  // A unit is (row tile, KV head, split); CTAs take units from an atomic
  // counter in the workspace until none are left.
  for (;;) {
    __syncthreads();
    if (tid == 0) {
      sh.unit = atomicAdd(p.unit_ctr, 1);
      sh.info[0] = -1;
    }
    __syncthreads();
    const int u = sh.unit;
    if (u >= p.n_units || sh.abort) break;
    const int split = u % p.S_p;
    const int g = (u / p.S_p) % p.H_kv;
    const int tile = u / (p.S_p * p.H_kv);
    if (warp == 0) tc::locate_tile(p, tile, NT * TT, sh.info);
    __syncthreads();
    const int d = sh.info[0];
    if (d < 0) continue;
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
    const int b_lo = tok0 / m;
    const int nbc = (tok0 + ntok - 1) / m - b_lo + 1;  // branches of this unit's rows

    // private lengths and packed page offsets of the unit's branches
    if (warp == 0) {
      int base = 0;
      for (int c0 = 0; c0 < nbc; c0 += 32) {
        const int bl = c0 + lane;
        int np = 0;
        if (bl < nbc) {
          int Lb = p.branch_len[b_lo + bl];
          const int cap = p.max_pages * kPage;
          if (Lb < 0 || Lb > cap) {
            flag_error(p.err, HPD_DEVERR_BRANCH_LEN);
            Lb = min(max(Lb, 0), cap);
          }
          sh.blen[bl] = Lb;
          np = ceil_div_i(Lb, kPage);
        }
        int incl = np;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int v = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += v;
        }
        if (bl < nbc) sh.page_start[bl] = base + incl - np;
        base += __shfl_sync(0xffffffffu, incl, 31);
      }
      if (lane == 0) sh.page_start[nbc] = base;
    }
    // prefix keys needed by the unit's rows (fork-position prefixes may be short)
    auto prefix_limit = [&](int r) -> int {
      if (r >= nrows) return 0;
      if (!p.branch_prefix_len) return P_d;
      const int b = (tok0 + r / G) / m;
      int f = p.branch_prefix_len[b];
      if (f < 0 || f > P_d) {
        flag_error(p.err, HPD_DEVERR_FORK_LEN);
        f = min(max(f, 0), P_d);
      }
      return f;
    };
    if (tid == 0) sh.kmax = p.branch_prefix_len ? 0 : P_d;
    __syncthreads();
    if (p.branch_prefix_len)
      for (int r = tid; r < NT * kRows; r += L::kThreads) atomicMax(&sh.kmax, prefix_limit(r));
    const int P_s = sh.page_start[nbc];
    // page ids of the packed suffix pages (valid ids only)
    auto page_lookup = [&](int gp) -> int {
      int lo = 0, hi = nbc;  // largest bl with page_start[bl] <= gp
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (sh.page_start[mid] <= gp) lo = mid; else hi = mid;
      }
      int pg = p.page_table[static_cast<size_t>(b_lo + lo) * p.max_pages + (gp - sh.page_start[lo])];
      if (pg < 0 || pg >= p.num_pages) {
        flag_error(p.err, HPD_DEVERR_PAGE_ID);
        pg = 0;
      }
      return pg;
    };
    for (int gp = tid; gp < min(P_s, kPageCap); gp += L::kThreads) page_tab[gp] = page_lookup(gp);
    __syncthreads();
    const int nP = ceil_div_i(sh.kmax, kBlk);               // prefix blocks
    const int nS = ceil_div_i(P_s, kPagesPerBlock);         // suffix blocks
    const int N = nP + nS;
    const int blk_lo = static_cast<int>(static_cast<long long>(split) * N / p.S_p);
    const int blk_hi = static_cast<int>(static_cast<long long>(split + 1) * N / p.S_p);
    const int n_blocks = blk_hi - blk_lo;
    const bool final_out = p.S_p == 1;

    // (token, head) index of unit row r; partial slot index for several splits
    auto pair_index = [&](int r) -> size_t {
      return static_cast<size_t>(tok0 + r / G) * p.H_q + g * G + r % G;
    };
    auto slot_index = [&](int r) -> size_t {
      return static_cast<size_t>(split) * p.rows_total * p.H_q + pair_index(r);
    };
    if (n_blocks <= 0) {
      for (int r = tid; r < nrows; r += L::kThreads) {
        if (final_out) {
          uint4 *o = reinterpret_cast<uint4 *>(p.out + pair_index(r) * D);
          for (int c = 0; c < D / 8; ++c) o[c] = make_uint4(0u, 0u, 0u, 0u);
          if (p.lse) p.lse[pair_index(r)] = NEG_INF;
        } else {
          p.l_part[slot_index(r)] = NEG_INF;
        }
      }
      continue;
    }

    if (warp == 0) {
      // ---------------------------------------------------- producer --
      // The whole warp runs this loop with warp-uniform values; one elected
      // lane issues each copy.
      if (uidx == 0 && lane == 0) {
        prefetch_tmap(&tm_q);
        prefetch_tmap(&tm_k);
        prefetch_tmap(&tm_v);
        prefetch_tmap(&tm_kc);
        prefetch_tmap(&tm_vc);
      }
      __syncwarp();
      mbar_arrive_expect_tx_elect(bar(sh.q_full), NT * L::kTileBytes);
      for (int t = 0; t < NT; ++t)
        for (int c = 0; c < L::kChunks; ++c)
          tma_load_3d_elect(sbase + L::kQ + t * L::kTileBytes + c * L::kChunkBytes, &tm_q,
                            bar(sh.q_full), c * 64, g * G, tok0 + t * TT);
      auto page_of = [&](int gp) { return gp < kPageCap ? page_tab[gp] : page_lookup(gp); };
      // one block of K (or V) into stage `dst`
      auto load_block = [&](int jb, uint32_t dst, uint32_t b, const CUtensorMap *prefix_map,
                            const CUtensorMap *page_map) {
        mbar_arrive_expect_tx_elect(b, L::kTileBytes);
        if (jb < nP) {
          for (int c = 0; c < L::kChunks; ++c)
            tma_load_3d_elect(dst + c * L::kChunkBytes, prefix_map, b, c * 64, g, pc0 + jb * kBlk);
        } else {
          const int gp0 = (jb - nP) * kPagesPerBlock;
          for (int i = 0; i < kPagesPerBlock; ++i) {
            // slots past the last page repeat it: finite values, never visible
            const int pg = page_of(min(gp0 + i, P_s - 1));
            for (int c = 0; c < L::kChunks; ++c)
              tma_load_4d_elect(dst + c * L::kChunkBytes + i * kPage * 128, page_map, b, c * 64, g,
                                0, pg);
          }
        }
      };
      auto wait_all = [&](uint64_t &b, int parity) {
        return __all_sync(0xffffffffu, !sh.abort && mbar_wait(bar(b), parity));
      };
      int issued_k = 0, issued_v = 0;
      for (int j = 0; j < n_blocks; ++j) {
        const int jg = jbase + j, s = jg & 1, prev = ((jg >> 1) - 1) & 1;
        if (jg >= 2 && !wait_all(sh.k_empty[s], prev)) {
          if (lane == 0) set_abort(sh, p.err);
          break;
        }
        load_block(blk_lo + j, sbase + L::kK + s * L::kTileBytes, bar(sh.k_full[s]), &tm_k,
                   &tm_kc);
        issued_k = j + 1;
        if (jg >= 2 && !wait_all(sh.v_empty[s], prev)) {
          if (lane == 0) set_abort(sh, p.err);
          break;
        }
        load_block(blk_lo + j, sbase + L::kV + s * L::kTileBytes, bar(sh.v_full[s]), &tm_v,
                   &tm_vc);
        issued_v = j + 1;
      }
      // Do not go on while a copy into this CTA's shared memory is in flight.
      mbar_wait(bar(sh.q_full), uidx & 1);
      for (int j = max(0, issued_k - 2); j < issued_k; ++j)
        mbar_wait(bar(sh.k_full[(jbase + j) & 1]), ((jbase + j) >> 1) & 1);
      for (int j = max(0, issued_v - 2); j < issued_v; ++j)
        mbar_wait(bar(sh.v_full[(jbase + j) & 1]), ((jbase + j) >> 1) & 1);
    } else if (warp == 1) {
      // ---------------------------------------------------- MMA issuer --
      // The whole warp runs this loop with warp-uniform values; one elected
      // lane issues each MMA / commit (see sm100.cuh).
      constexpr uint32_t idesc_qk = idesc_bf16_f32(kRows, kBlk, false);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(kRows, D, true);
      // Shared-memory descriptors: a tile / stage / k-step offset only adds
      // (offset >> 4) to the start-address field (bits 0-13), which cannot
      // carry: every address stays below 256 KB.
      const uint64_t dq0 = smem_desc_sw128(sbase + L::kQ, 16, 1024);
      const uint64_t dk0 = smem_desc_sw128(sbase + L::kK, 16, 1024);
      // S[col] = Q_t K^T of global block jg
      auto issue_qk = [&](int t, int jg, uint32_t col) {
        const uint64_t qd = dq0 + ((t * L::kTileBytes) >> 4);
        const uint64_t kd = dk0 + (((jg & 1) * L::kTileBytes) >> 4);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = ((kk >> 2) * L::kChunkBytes + (kk & 3) * 32) >> 4;
          mma_ss(tmem + col, qd + off, kd + off, idesc_qk, kk > 0);
        }
      };
      // O_t (+)= P V of global block jg, P in TMEM at column pcol: one N = D
      // MMA per 16 keys.  V is MN-major (D contiguous): 64-column swizzle
      // atoms kChunkBytes apart along N (leading byte offset), 8-key groups
      // 1024 bytes apart along K (stride byte offset).
      const uint64_t dv0 = smem_desc_sw128(sbase + L::kV, L::kChunkBytes, 1024);
      auto issue_pv = [&](int t, int jg, bool first, uint32_t pcol) {
        const uint64_t vd = dv0 + (((jg & 1) * L::kTileBytes) >> 4);
#pragma unroll
        for (int kk = 0; kk < kBlk / 16; ++kk)
          mma_ts(tmem + L::col_o(t), tmem + pcol + kk * 8, vd + ((kk * 16 * 128) >> 4), idesc_pv,
                 (!first || kk > 0) ? 1u : 0u);
      };
      auto wait = [&](uint64_t &b, int parity) {
        if (!__all_sync(0xffffffffu, !sh.abort && mbar_wait(bar(b), parity))) return false;
        tc_fence_after();
        return true;
      };
      bool ok = wait(sh.q_full, uidx & 1);
      if constexpr (NT == 1) {
        for (int j = 0; ok && j <= n_blocks; ++j) {
          if (j < n_blocks) {
            const int jg = jbase + j, s = jg & 1;
            if (!(ok = wait(sh.k_full[s], (jg >> 1) & 1))) break;
            issue_qk(0, jg, L::col_s(s));
            mma_commit(bar(sh.s_full[s]));
            mma_commit(bar(sh.k_empty[s]));
          }
          if (j >= 1) {
            const int jg = jbase + j - 1, s = jg & 1;
            if (!(ok = wait(sh.p_full[s], (jg >> 1) & 1) && wait(sh.v_full[s], (jg >> 1) & 1)))
              break;
            issue_pv(0, jg, j == 1, L::col_s(s));
            mma_commit(bar(sh.pv_done[0]));
            mma_commit(bar(sh.v_empty[s]));
          }
        }
      } else {
        // tile t's S lives at col_s(t); tiles alternate on the tensor pipe:
        //   PV_0(j)  QK_0(j+1)  PV_1(j)  QK_1(j+1)  ...
        if (ok && (ok = wait(sh.k_full[jbase & 1], (jbase >> 1) & 1))) {
          for (int t = 0; t < n_act; ++t) {
            issue_qk(t, jbase, L::col_s(t));
            mma_commit(bar(sh.s_full[t]));
          }
          mma_commit(bar(sh.k_empty[jbase & 1]));
        }
        for (int j = 0; ok && j < n_blocks; ++j) {
          const int jg = jbase + j, s = jg & 1;
          const bool more = j + 1 < n_blocks;
          for (int t = 0; t < n_act; ++t) {
            if (!(ok = wait(sh.p_full[t], (jt[t] + j) & 1))) break;
            if (t == 0 && !(ok = wait(sh.v_full[s], (jg >> 1) & 1))) break;
            issue_pv(t, jg, j == 0, L::col_s(t));
            mma_commit(bar(sh.pv_done[t]));
            if (more) {
              if (t == 0 && !(ok = wait(sh.k_full[s ^ 1], ((jg + 1) >> 1) & 1))) break;
              issue_qk(t, jg + 1, L::col_s(t));
              mma_commit(bar(sh.s_full[t]));
            }
          }
          if (!ok) break;
          mma_commit(bar(sh.v_empty[s]));
          if (more) mma_commit(bar(sh.k_empty[s ^ 1]));
        }
      }
      if (!ok && lane == 0) set_abort(sh, p.err);
    } else {
      // ----------------------------------------------------- softmax --
      // Two warpgroups per row tile: warpgroup half h owns key columns
      // [64 h, 64 h + 64) of every block and output columns [64 h, 64 h + 64).
      constexpr int kH = L::kHalves;
      const int t = (warp - 2) / (4 * kH);            // row tile
      const int h = kH == 2 ? ((warp - 2) >> 2) & 1 : 0;  // column half
      const int quad = warp & 3;            // TMEM lane quadrant this warp may access
      const int r_in = quad * 32 + lane;    // row within the tile
      const int row = t * kRows + r_in;
      const uint32_t t_lane = tmem + (static_cast<uint32_t>(quad * 32) << 16);
      const uint32_t o_col = L::col_o(t) + h * (D / kH);
      const int cnt = NT == 1 ? jbase : jt[t];  // pv_done[t] phases completed before this unit
      auto tile_sync = [&]() {
        if (kH == 2) asm volatile("bar.sync %0, %1;" ::"r"(1 + t), "r"(256) : "memory");
      };
      if (t < n_act) {
        // the row's visible keys: prefix below lim_p; own branch's private
        // keys j <= last, which start at packed page ps
        const bool valid = row < nrows;
        const int token = tok0 + row / G;
        const int bl = valid ? token / m - b_lo : 0;
        const int lim_p = prefix_limit(row);
        const int ps = valid ? sh.page_start[bl] : 0;
        const int last = valid ? sh.blen[bl] - m + (token - (b_lo + bl) * m) : -1;
        const float sl2 = p.scale_log2;
        float m_run = NEG_INF, l_half = 0.f;
        bool ok = true;
        for (int j = 0; j < n_blocks; ++j) {
          const int jg = jbase + j;
          const int si = NT == 1 ? (jg & 1) : t;  // S buffer / barrier index
          const int ph = NT == 1 ? ((jg >> 1) & 1) : ((jt[t] + j) & 1);
          const uint32_t s_col = L::col_s(si);
          // warp-uniform outcome: the tcgen05.ld / st below are warp-collective
          if (!__all_sync(0xffffffffu, !sh.abort && mbar_wait(bar(sh.s_full[si]), ph))) {
            ok = false;
            break;
          }
          tc_fence_after();
          const int jb = blk_lo + j;
          int lo, hi;
          if (jb < nP) {
            lo = 0;
            hi = lim_p - jb * kBlk;
          } else {
            const int off = (ps - (jb - nP) * kPagesPerBlock) * kPage;  // column of own key 0
            lo = max(0, off);
            hi = min(kBlk, off + last + 1);
          }
          const int par = j & 1;
          auto xchg = [&](float mx) {
            sh.xmax[h][par][r_in] = mx;
            tile_sync();
            return fmaxf(mx, sh.xmax[h ^ 1][par][r_in]);
          };
          const float alpha =
              kH == 2 ? tc::softmax_half_tmem(t_lane + s_col, h, lo, hi, sl2, m_run, l_half, xchg)
                      : tc::softmax_block_tmem(t_lane + s_col, lo, hi, sl2, m_run, l_half);
          // Before O may be rescaled, the P V MMA of block j-1 must have
          // landed.  NT = 2: this tile's S commit was issued after that MMA,
          // and a commit fires only once every earlier MMA of the issuing
          // thread has completed, so it has.  NT = 1: P V (j-1) is issued
          // after Q K^T (j), so a warp that rescales waits for it.  Warps
          // skip the wait when they do not rescale, yet the parity test stays
          // exact: Q K^T (j) was issued after P V (j-2), so the S commit
          // awaited above implies P V (j-2) has completed, and P V (j) needs
          // this block's P; the barrier is in one of two consecutive phases.
          // The last block always waits, which gives the epilogue that bound.
          const bool rescale = __any_sync(0xffffffffu, j > 0 && alpha != 1.f);
          if (NT == 1 && j > 0 && (rescale || j == n_blocks - 1) &&
              !__all_sync(0xffffffffu, mbar_wait(bar(sh.pv_done[t]), (cnt + j - 1) & 1))) {
            ok = false;
            break;
          }
          // Rescale this half's O columns if any row of this warp needs it.
          if (rescale) {
            tc_fence_after();
#pragma unroll
            for (int c = 0; c < D / kH; c += 32) {
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
        if (!ok && lane == 0) set_abort(sh, p.err);
        // ------------------------------------------------ epilogue --
        // row sum over both halves (both halves reach this point together:
        // on a timeout, every wait of the tile's warps gives up)
        float l_run = l_half;
        if (kH == 2) {
          sh.xsum[h][r_in] = l_half;
          tile_sync();
          l_run += sh.xsum[h ^ 1][r_in];
        }
        // pv_done[t] has completed at least cnt + n_blocks - 1 phases (see
        // above), so the parity wait for the unit's last block is exact.
        if (ok && __all_sync(0xffffffffu,
                             mbar_wait(bar(sh.pv_done[t]), (cnt + n_blocks - 1) & 1))) {
          tc_fence_after();
          const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
          const float lse = l_run > 0.f ? (m_run + __log2f(l_run)) * kLn2 : NEG_INF;
#pragma unroll
          for (int c = 0; c < D / kH; c += 32) {
            uint32_t o[32];
            tmem_ld32(t_lane + o_col + c, o);
            tmem_ld_wait();
            if (!valid) continue;
            const int dc = h * (D / kH) + c;  // output column
            if (final_out) {
              uint4 *dst = reinterpret_cast<uint4 *>(p.out + pair_index(row) * D + dc);
#pragma unroll
              for (int e = 0; e < 32; e += 8)
                dst[e / 8] = make_uint4(
                    pack_bf16x2(__uint_as_float(o[e]) * inv, __uint_as_float(o[e + 1]) * inv),
                    pack_bf16x2(__uint_as_float(o[e + 2]) * inv, __uint_as_float(o[e + 3]) * inv),
                    pack_bf16x2(__uint_as_float(o[e + 4]) * inv, __uint_as_float(o[e + 5]) * inv),
                    pack_bf16x2(__uint_as_float(o[e + 6]) * inv, __uint_as_float(o[e + 7]) * inv));
            } else {
              float *dst = p.o_part + slot_index(row) * D + dc;
#pragma unroll
              for (int e = 0; e < 32; e += 4)
                *reinterpret_cast<float4 *>(dst + e) =
                    make_float4(__uint_as_float(o[e]) * inv, __uint_as_float(o[e + 1]) * inv,
                                __uint_as_float(o[e + 2]) * inv, __uint_as_float(o[e + 3]) * inv);
            }
          }
          if (valid && h == 0) {
            if (final_out) {
              if (p.lse) p.lse[pair_index(row)] = lse;
            } else {
              p.l_part[slot_index(row)] = lse;
            }
          }
          tc_fence_before();  // O is read before the next unit's MMAs overwrite it
        } else if (ok && lane == 0) {
          set_abort(sh, p.err);
        }
      }
    }
    // end of unit: every role is done with Q / K / V and with O in TMEM
    jbase += n_blocks;
    if (NT == 2) {
      jt[0] += n_blocks;
      if (n_act == 2) jt[1] += n_blocks;
    }
    ++uidx;
  }

  // ------------------------------------------------------------ teardown --
  // every MMA issued by this CTA has finished before TMEM is released
  if (warp == 1) {
    mma_commit(bar(sh.mma_done));
    mbar_wait(bar(sh.mma_done), 0);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
  // the last CTA to finish resets the unit counters for the next call
  if (tid == 0) {
    __threadfence();
    if (atomicAdd(p.unit_ctr + 1, 1) == static_cast<int>(gridDim.x) - 1) {
      atomicExch(p.unit_ctr, 0);
      atomicExch(p.unit_ctr + 1, 0);
    }
  }
}

template <int D, int NT>
cudaError_t launch_tc(const AttnParams &p, const Plan &plan, cudaStream_t s) {
  using L = TcLayout<D, NT>;
  CUtensorMap tq, tk, tv, tkc, tvc;
  cudaError_t e = tc::make_prefix_maps(p, &tq, &tk, &tv);
  if (e == cudaSuccess) e = tc::make_page_map(&tkc, p.k_cache, D, p.H_kv, p.num_pages);
  if (e == cudaSuccess) e = tc::make_page_map(&tvc, p.v_cache, D, p.H_kv, p.num_pages);
  if (e != cudaSuccess) return e;
  static std::atomic<uint64_t> configured{0};
  int dev = 0;
  e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(configured.load(std::memory_order_acquire) & bit)) {
    e = cudaFuncSetAttribute(branch_attn_tc_kernel<D, NT>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(L::kDynSmem));
    if (e != cudaSuccess) return e;
    configured.fetch_or(bit, std::memory_order_acq_rel);
  }
  static int sms[64] = {0};
  if (sms[dev & 63] == 0) {
    int n = 0;
    e = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    sms[dev & 63] = n;
  }
  const int n_units = p.n_units;
  const dim3 grid(static_cast<unsigned>(std::min(n_units, sms[dev & 63])), 1, 1);
  branch_attn_tc_kernel<D, NT><<<grid, L::kThreads, L::kDynSmem, s>>>(tq, tk, tv, tkc, tvc, p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_branch_attn_tc(const AttnParams &p, const Plan &plan, cudaStream_t s) {
  if (plan.tiles_max <= 0) return cudaSuccess;
  if (plan.tc_tiles == 2)
    return p.D == 64 ? launch_tc<64, 2>(p, plan, s) : launch_tc<128, 2>(p, plan, s);
  return p.D == 64 ? launch_tc<64, 1>(p, plan, s) : launch_tc<128, 1>(p, plan, s);
}

}  // namespace hpd
