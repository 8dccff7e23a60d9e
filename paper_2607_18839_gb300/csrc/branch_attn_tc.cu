// branch_attn_tc.cu -- the branch-attention step on 5th-generation tensor
// cores: shared prefix and private suffixes in one persistent kernel.
//
// What it computes (Sec. 3.3, "Dynamic Branch Forking and Efficient Context
// Isolation"; Sec. 3.4 for the m P-MTP queries): all query rows of a page's
// branches that read KV head g are stacked (row r <-> token
// branch_cu[d]*m + r/G, query head g*G + r%G).  Each row attends to
//   - the page's shared prefix keys [0, P_b), P_b its branch's fork-position
//     prefix length (P_d when none is given), and
//   - its own branch's private keys j <= L_b - m + i (i = the row's query).
// The page's prefix is read once per 128 stacked rows instead of once per
// branch: that is the shared-prefix KV reuse the method relies on.
//
// Key blocks: a unit walks 128-key blocks of two kinds,
//   prefix blocks  128 consecutive prefix keys: one 3-D TMA box per 64
//                  columns from the contiguous prefix, or, with a paged
//                  prefix, 8 pool pages of 16 keys from the page's prefix
//                  page table (Algorithm 1: forks share the parent's pages),
//   suffix blocks  8 pages of 16 keys, packed from the private caches of the
//                  unit's branches in branch order.
// A paged block whose 8 pages are consecutive pool pages loads as one 8-page
// 4-D box per 64 columns, else as one box per page.
// For every row and block the visible columns form one interval [lo, hi):
// a prefix block's keys below the row's limit, or the row's own branch's
// pages up to its causal bound.  Rows of other branches see nothing of a
// suffix page, so their probabilities are zero there.
//
// Work units: (row tile of 128 stacked rows, KV head, split), a split being
// an even share of the tile's blocks.  One CTA per SM takes units from an
// atomic counter, and its roles run one unit apart so that nothing drains
// between units:
//   warp 10     scheduler: takes the next unit and prepares its metadata
//               (page, rows, private lengths, fork limits, packed page ids)
//               in one of two shared-memory slots while the other is in use.
//   warps 0, 11 TMA producers: warp 0 the unit's Q tile and then its K
//               blocks, warp 11 its V blocks, each into a three-stage ring
//               (128-byte swizzle); a K stage is refilled as soon as its Q
//               K^T (or Q copy) is done, whatever the V ring waits for.
//   warp 1      TMEM owner and MMA issuer: copies each unit's Q tile from
//               its K stage into TMEM (tcgen05.cp, double buffered by unit),
//               then one global sequence of blocks across units, in the
//               order QK(b), PV(b-1):
//                 S = Q K^T   Q read from TMEM, K from shared memory; S into
//                             TMEM (fp32, double buffered by block)
//                 O += P V    P read from TMEM (bf16, written over S), V from
//                             shared memory; O accumulated in TMEM
//               With both A operands in TMEM, shared memory serves only K,
//               V and their TMA writes (its bandwidth is the scarce port).
//   warps 2..9  softmax: two warpgroups, each owning half of every block's
//               128 key columns and half of O's columns; thread t of warp w
//               owns TMEM lane 32*(w%4)+t, i.e. one query row.  The two
//               halves of a row exchange their partial max through shared
//               memory.  O is rescaled in TMEM only when a row's running
//               max grows by more than 2^8; the stale max stays exact after
//               the final normalisation.  At a unit change they only read
//               the next unit's metadata before the epilogue.
// One split: the unit writes the final bf16 output and lse.  Several splits:
// it writes its normalised fp32 partial and lse for merge.cu.
// All waits are bounded; a timeout sets HPD_DEVERR_TIMEOUT, every role
// leaves its loop, and the CTA drains its in-flight copies and MMAs, frees
// its TMEM and exits.  No role waits on a hardware barrier (bar.sync) inside
// its loop, so a role that leaves early cannot strand another.
#include <algorithm>
#include <atomic>

#include "tc_common.cuh"

namespace hpd {
namespace {

using namespace sm100;
using tc::kBlk;
using tc::kRows;

constexpr uint32_t kTmemCols = 512;
constexpr int kMaxUnitBranches = kRows + 1;  // branches touching 128 stacked rows
constexpr int kPageCap = 2048;               // suffix page ids kept in shared memory
constexpr int kPagesPerBlock = kBlk / kPage;
constexpr int kSoftmaxWarps = 8;
constexpr int kSchedWarp = 2 + kSoftmaxWarps;
constexpr int kVWarp = kSchedWarp + 1;
constexpr int kThreads = 32 * (kVWarp + 1);
// consumers of a metadata slot: two producers, MMA issuer, softmax warps
constexpr uint32_t kMetaConsumers = 3 + kSoftmaxWarps;
constexpr int kMaxRing = 3;  // largest K / V ring

// Metadata of one unit, written by the scheduler warp.
struct UnitMeta {
  int valid;     // 0: no units left
  int g;         // KV head
  int split;     // split index
  int tok0;      // first query token of the tile
  int nrows;     // stacked rows (ntok * G)
  int b_lo;      // first branch
  int nbc;       // branches of the rows
  int nP;        // prefix blocks
  int pc0;       // first prefix token of the page
  int blk_lo;    // first block of the split
  int n_blocks;  // blocks of the split (> 0)
  int doc;       // page (document) of the tile
  int pp_last;   // paged prefix: last prefix page any row of the tile sees
  int page_start[kMaxUnitBranches + 1];  // packed page offset of each branch
  int blen[kMaxUnitBranches];            // private length L_b (clamped)
  int fork[kMaxUnitBranches];            // prefix keys visible to the branch
  int page_tab[kPageCap];                // packed suffix page ids
};

template <int D>
struct TcLayout {
  static constexpr int kChunks = D / 64;                // 64-column (128-byte) boxes
  static constexpr uint32_t kChunkBytes = kRows * 128;  // 128 rows x 128 bytes
  static constexpr uint32_t kTileBytes = kChunks * kChunkBytes;
  static constexpr int kKStages = 3, kVStages = 3;
  static constexpr uint32_t kK = 0;
  static constexpr uint32_t kV = kK + kKStages * kTileBytes;
  static constexpr uint32_t kMeta = kV + kVStages * kTileBytes;  // 2 UnitMeta slots
  static constexpr uint32_t kBytes = kMeta + 2 * sizeof(UnitMeta);
  static constexpr uint32_t kDynSmem = kBytes + 1024;   // slack to align to 1024
  // TMEM columns: S of block buffer i at col_s(i), O at kColO, the Q rows of
  // unit slot u at col_q(u) (D / 2 columns: two bf16 per column)
  static constexpr uint32_t kColO = 256;
  static __device__ __forceinline__ uint32_t col_s(int i) { return i ? 128u : 0u; }
  static __device__ __forceinline__ uint32_t col_q(int u) { return u ? 448u : 384u; }
};

struct __align__(8) TcShared {
  uint64_t meta_full[2], meta_empty[2];
  uint64_t k_full[kMaxRing], v_full[kMaxRing];
  uint64_t k_empty[kMaxRing], v_empty[kMaxRing];
  uint64_t s_full[2], p_full[2];  // per S buffer
  uint64_t pv_done;
  uint64_t o_full, o_empty;
  uint64_t mma_done;
  uint32_t tmem_base;
  int abort;
  // the two column halves of a row exchange their partial row max (double
  // buffered by block parity) and, at the end of a unit, their partial sums;
  // seq counters publish each value ([half][TMEM lane quadrant])
  float xmax[2][2][kRows];  // [half][block parity][row]
  float xsum[2][kRows];     // [half][row]
  int xseq[2][2][4];        // [max | sum][half][quadrant]
};

__device__ __forceinline__ void set_abort(TcShared &sh, uint32_t *err) {
  atomicExch(&sh.abort, 1);
  flag_error(err, HPD_DEVERR_TIMEOUT);
}
__device__ __forceinline__ bool aborted(const TcShared &sh) {
  return *reinterpret_cast<const volatile int *>(&sh.abort) != 0;
}

// Publish `seq` at *flag after this warp's earlier shared-memory writes
// (release store by lane 0 once the warp's lanes are ordered by __syncwarp).
__device__ __forceinline__ void publish_seq(int *flag, int seq) {
  __syncwarp();
  if ((threadIdx.x & 31) == 0)
    asm volatile("st.release.cta.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(flag)), "r"(seq)
                 : "memory");
}
__device__ __forceinline__ int load_seq(const int *flag) {
  int v;
  asm volatile("ld.acquire.cta.shared::cta.b32 %0, [%1];" : "=r"(v) : "r"(smem_u32(flag)) : "memory");
  return v;
}
// Slow path of await_seq, out of line so that the clock read stays off the
// fast path.
__device__ __noinline__ bool await_seq_slow(const int *flag, int seq, const int *abort) {
  const uint64_t t0 = globaltimer();
  for (uint32_t i = 1; load_seq(flag) < seq; ++i)
    if ((i & 63u) == 0 &&
        (*reinterpret_cast<const volatile int *>(abort) || globaltimer() - t0 > kWaitLimitNs))
      return false;
  return true;
}
// Wait (bounded) until *flag >= seq, with acquire ordering; false on timeout
// or abort.
__device__ __forceinline__ bool await_seq(const int *flag, int seq, const TcShared &sh) {
  return load_seq(flag) >= seq || await_seq_slow(flag, seq, &sh.abort);
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    branch_attn_tc_kernel(const __grid_constant__ CUtensorMap tm_k,
                          const __grid_constant__ CUtensorMap tm_v,
                          const __grid_constant__ CUtensorMap tm_kc,
                          const __grid_constant__ CUtensorMap tm_vc,
                          const __grid_constant__ CUtensorMap tm_k8,
                          const __grid_constant__ CUtensorMap tm_v8,
                          const __grid_constant__ CUtensorMap tm_q, const AttnParams p) {
  using L = TcLayout<D>;
  extern __shared__ uint8_t smem_raw[];
  __shared__ TcShared sh;
  const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
  UnitMeta *meta =
      reinterpret_cast<UnitMeta *>(smem_raw + (sbase - smem_u32(smem_raw)) + L::kMeta);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = p.G, m = p.m;
  const int TT = kRows / G;  // tokens per 128-row tile
  const float NEG_INF = -__int_as_float(0x7f800000);
  auto bar = [](uint64_t &b) { return smem_u32(&b); };
  // bounded wait on an mbarrier phase, warp-uniform outcome; false on abort
  auto wait_bar = [&](uint64_t &b, int parity) {
    return __all_sync(0xffffffffu, mbar_wait(bar(b), parity, &sh.abort));
  };

  // ------------------------------------------------------ once per CTA --
  if (tid == 0) {
    sh.abort = 0;
    for (int s = 0; s < kMaxRing; ++s) {
      mbar_init(bar(sh.k_full[s]), 1);
      mbar_init(bar(sh.v_full[s]), 1);
      mbar_init(bar(sh.k_empty[s]), 1);
      mbar_init(bar(sh.v_empty[s]), 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(bar(sh.meta_full[s]), 1);
      mbar_init(bar(sh.meta_empty[s]), kMetaConsumers);
      mbar_init(bar(sh.s_full[s]), 1);
      mbar_init(bar(sh.p_full[s]), kSoftmaxWarps);
    }
    mbar_init(bar(sh.pv_done), 1);
    mbar_init(bar(sh.o_full), 1);
    mbar_init(bar(sh.o_empty), kSoftmaxWarps);
    mbar_init(bar(sh.mma_done), 1);
    fence_mbar_init();
  }
  if (tid < 16) (&sh.xseq[0][0][0])[tid] = 0;
  if (warp == 1) {
    tmem_alloc(smem_u32(&sh.tmem_base), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sh.tmem_base;
  pdl_wait();     // the unit order (and everything before it) is complete
  pdl_trigger();  // the merge of the splits may launch; it waits for this grid

  if (warp == kSchedWarp) {
    // ------------------------------------------------------- scheduler --
    // Fills slot k & 1 with the k-th unit of this CTA that has keys; units
    // without any get their output written here and are skipped.
    for (int k = 0;; ++k) {
      const int slot = k & 1;
      if (k >= 2 && !wait_bar(sh.meta_empty[slot], ((k >> 1) - 1) & 1)) {
        if (lane == 0) set_abort(sh, p.err);
        break;
      }
      UnitMeta &M = meta[slot];
      bool have = false;
      for (;;) {
        int u = 0;
        if (lane == 0) u = atomicAdd(p.unit_ctr, 1);
        u = __shfl_sync(0xffffffffu, u, 0);
        if (u >= p.n_units || aborted(sh)) break;
        if (p.unit_order) u = p.unit_order[u];  // longest units first
        const int split = u % p.S_p;
        const int g = (u / p.S_p) % p.H_kv;
        const int tile = u / (p.S_p * p.H_kv);
        // the page owning the tile: page d has ceil(#branches(d) * m / TT) tiles
        int d = -1, lt = 0, b0 = 0, b1 = 0;
        for (int d0 = 0, base = 0; d0 < p.n_docs && base <= tile; d0 += 32) {
          const int dd = d0 + lane;
          int tiles = 0, c0 = 0, c1 = 0;
          if (dd < p.n_docs) {
            c0 = min(max(p.branch_cu[dd], 0), p.B);
            c1 = min(max(p.branch_cu[dd + 1], 0), p.B);
            if (c1 < c0) {
              flag_error(p.err, HPD_DEVERR_BRANCH_CU);
              c1 = c0;
            }
            tiles = ceil_div_i((c1 - c0) * m, TT);
          }
          int incl = tiles;
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += v;
          }
          const int excl = incl - tiles;
          const unsigned hit =
              __ballot_sync(0xffffffffu, tiles > 0 && tile >= base + excl && tile < base + incl);
          if (hit) {
            const int src = __ffs(hit) - 1;
            d = __shfl_sync(0xffffffffu, dd, src);
            lt = __shfl_sync(0xffffffffu, tile - base - excl, src);
            b0 = __shfl_sync(0xffffffffu, c0, src);
            b1 = __shfl_sync(0xffffffffu, c1, src);
            break;
          }
          base += __shfl_sync(0xffffffffu, incl, 31);
        }
        if (d < 0) continue;
        int pc0, P_d;
        bool bad_prefix;
        page_prefix(p, d, pc0, P_d, bad_prefix);
        if (lane == 0 && bad_prefix) flag_error(p.err, HPD_DEVERR_PREFIX_CU);
        const int tok0 = b0 * m + lt * TT;
        const int ntok = min(TT, (b1 - b0) * m - lt * TT);
        const int b_lo = tok0 / m;
        const int nbc = (tok0 + ntok - 1) / m - b_lo + 1;
        // private lengths, packed page offsets and fork limits of the branches
        int base = 0, kmax = 0;
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
            int f = P_d;
            if (p.branch_prefix_len) {
              f = p.branch_prefix_len[b_lo + bl];
              if (f < 0 || f > P_d) {
                flag_error(p.err, HPD_DEVERR_FORK_LEN);
                f = min(max(f, 0), P_d);
              }
            }
            M.blen[bl] = Lb;
            M.fork[bl] = f;
            kmax = max(kmax, f);
            np = ceil_div_i(Lb, kPage);
          }
          int incl = np;
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += v;
          }
          if (bl < nbc) M.page_start[bl] = base + incl - np;
          base += __shfl_sync(0xffffffffu, incl, 31);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) kmax = max(kmax, __shfl_xor_sync(0xffffffffu, kmax, o));
        const int P_s = base;
        if (lane == 0) M.page_start[nbc] = P_s;
        __syncwarp();
        // packed suffix page ids (valid ids only), four lookups in flight
        const int n_tab = min(P_s, kPageCap);
        for (int gp0 = 0; gp0 < n_tab; gp0 += 128) {
          int addr[4];
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const int gp = gp0 + q * 32 + lane;
            addr[q] = -1;
            if (gp < n_tab) {
              int lo = 0, hi = nbc;  // largest bl with page_start[bl] <= gp
              while (hi - lo > 1) {
                const int mid = (lo + hi) >> 1;
                if (M.page_start[mid] <= gp) lo = mid; else hi = mid;
              }
              addr[q] = (b_lo + lo) * p.max_pages + (gp - M.page_start[lo]);
            }
          }
          int pg[4];
#pragma unroll
          for (int q = 0; q < 4; ++q) pg[q] = addr[q] >= 0 ? p.page_table[addr[q]] : 0;
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            if (addr[q] < 0) continue;
            if (pg[q] < 0 || pg[q] >= p.num_pages) {
              flag_error(p.err, HPD_DEVERR_PAGE_ID);
              pg[q] = 0;
            }
            M.page_tab[gp0 + q * 32 + lane] = pg[q];
          }
        }
        const int N = ceil_div_i(kmax, kBlk) + ceil_div_i(P_s, kPagesPerBlock);
        const int blk_lo = static_cast<int>(static_cast<long long>(split) * N / p.S_p);
        const int blk_hi = static_cast<int>(static_cast<long long>(split + 1) * N / p.S_p);
        const int nrows = ntok * G;
        if (blk_hi <= blk_lo) {
          // no key in this split: zero output (one split) or an empty partial
          for (int r = lane; r < nrows; r += 32) {
            const size_t pair = static_cast<size_t>(tok0 + r / G) * p.H_q + g * G + r % G;
            if (p.S_p == 1) {
              uint4 *o = reinterpret_cast<uint4 *>(p.out + pair * D);
              for (int c = 0; c < D / 8; ++c) o[c] = make_uint4(0u, 0u, 0u, 0u);
              if (p.lse) p.lse[pair] = NEG_INF;
            } else {
              p.l_part[static_cast<size_t>(split) * p.rows_total * p.H_q + pair] = NEG_INF;
            }
          }
          continue;
        }
        if (lane == 0) {
          M.g = g;
          M.split = split;
          M.tok0 = tok0;
          M.nrows = nrows;
          M.b_lo = b_lo;
          M.nbc = nbc;
          M.nP = ceil_div_i(kmax, kBlk);
          M.pc0 = pc0;
          M.doc = d;
          M.pp_last = max(kmax - 1, 0) / kPage;
          M.blk_lo = blk_lo;
          M.n_blocks = blk_hi - blk_lo;
        }
        have = true;
        break;
      }
      if (lane == 0) M.valid = have ? 1 : 0;
      __syncwarp();
      __threadfence_block();
      if (lane == 0) mbar_arrive(bar(sh.meta_full[slot]));
      if (!have) break;
    }
  } else if (warp == 0 || warp == kVWarp) {
    // ------------------------------------------------------- producers --
    // The whole warp runs this loop with warp-uniform values; one elected
    // lane issues each copy.  Warp 0: Q and K; warp kVWarp: V.  The K ring
    // carries each unit's Q tile ahead of its K blocks: ring entry jbase + k
    // is unit k's Q, entry jg + k + 1 the K of global block jg.
    const bool is_k = warp == 0;
    if (lane == 0) {
      prefetch_tmap(&tm_q);
      prefetch_tmap(&tm_k);
      prefetch_tmap(&tm_v);
      prefetch_tmap(&tm_kc);
      prefetch_tmap(&tm_vc);
      prefetch_tmap(&tm_k8);
      prefetch_tmap(&tm_v8);
    }
    __syncwarp();
    int jbase = 0, issued_k = 0, issued_v = 0;
    bool ok = true;
    for (int k = 0; ok; ++k) {
      const int slot = k & 1;
      if (!(ok = wait_bar(sh.meta_full[slot], (k >> 1) & 1))) break;
      const UnitMeta &M = meta[slot];
      if (!M.valid) break;
      const int g = M.g, nP = M.nP, pc0 = M.pc0, blk_lo = M.blk_lo, nb = M.n_blocks;
      const int P_s = M.page_start[M.nbc];
      // page id of packed suffix page gp (past the shared-memory table: looked
      // up again; an id out of range was flagged by the scheduler)
      auto page_of = [&](int gp) -> int {
        if (gp < kPageCap) return M.page_tab[gp];
        int lo = 0, hi = M.nbc;
        while (hi - lo > 1) {
          const int mid = (lo + hi) >> 1;
          if (M.page_start[mid] <= gp) lo = mid; else hi = mid;
        }
        const int pg = p.page_table[static_cast<size_t>(M.b_lo + lo) * p.max_pages +
                                    (gp - M.page_start[lo])];
        if (pg < 0 || pg >= p.num_pages) {
          flag_error(p.err, HPD_DEVERR_PAGE_ID);
          return 0;
        }
        return pg;
      };
      // paged prefix: lane i < 8 fetches the pool page of prefix page
      // 8 jb + i (pages past the last one any row sees repeat it: finite
      // values, never visible); called before waiting for the ring slot so
      // the lookup overlaps the wait
      const bool paged_prefix = p.prefix_page_table != nullptr;
      auto prefix_pid = [&](int jb) -> int {
        if (!paged_prefix || jb >= nP || lane >= kPagesPerBlock) return 0;
        return prefix_page(p, M.doc, min(jb * kPagesPerBlock + lane, M.pp_last));
      };
      // one block of K (or V) into stage `dst`.  A paged block is 8 pages
      // (lane i < 8 holds page i); when they are consecutive pool pages one
      // 8-page box loads them all, else one box per page.
      auto load_block = [&](int jb, int pid, uint32_t dst, uint32_t b,
                            const CUtensorMap *prefix_map, const CUtensorMap *page_map,
                            const CUtensorMap *run_map) {
        mbar_arrive_expect_tx_elect(b, L::kTileBytes);
        if (jb < nP && !paged_prefix) {
          for (int c = 0; c < L::kChunks; ++c)
            tma_load_3d_elect(dst + c * L::kChunkBytes, prefix_map, b, c * 64, g, pc0 + jb * kBlk);
          return;
        }
        int pg = pid;
        if (jb >= nP && lane < kPagesPerBlock)  // slots past the last page repeat it
          pg = page_of(min((jb - nP) * kPagesPerBlock + lane, P_s - 1));
        const int next = __shfl_down_sync(0xffffffffu, pg, 1);
        const unsigned run =
            __ballot_sync(0xffffffffu, lane < kPagesPerBlock - 1 && next == pg + 1);
        if (p.num_pages >= kPagesPerBlock && (run & 0x7fu) == 0x7fu) {
          const int pg0 = __shfl_sync(0xffffffffu, pg, 0);
          for (int c = 0; c < L::kChunks; ++c)
            tma_load_4d_elect(dst + c * L::kChunkBytes, run_map, b, c * 64, g, 0, pg0);
        } else {
          for (int i = 0; i < kPagesPerBlock; ++i) {
            const int pgi = __shfl_sync(0xffffffffu, pg, i);
            for (int c = 0; c < L::kChunks; ++c)
              tma_load_4d_elect(dst + c * L::kChunkBytes + i * kPage * 128, page_map, b, c * 64, g,
                                0, pgi);
          }
        }
      };
      if (is_k) {  // the unit's Q tile: tokens [tok0, tok0 + 128 / G), heads of KV head g
        const int e = jbase + k, s = e % L::kKStages;
        if (e >= L::kKStages && !(ok = wait_bar(sh.k_empty[s], ((e / L::kKStages) - 1) & 1)))
          break;
        mbar_arrive_expect_tx_elect(bar(sh.k_full[s]), L::kTileBytes);
        for (int c = 0; c < L::kChunks; ++c)
          tma_load_3d_elect(sbase + L::kK + s * L::kTileBytes + c * L::kChunkBytes, &tm_q,
                            bar(sh.k_full[s]), c * 64, g * G, M.tok0);
        issued_k = e + 1;
      }
      for (int j = 0; j < nb; ++j) {
        const int jg = jbase + j;
        const int pid = prefix_pid(blk_lo + j);
        if (is_k) {
          const int e = jg + k + 1, s = e % L::kKStages;
          if (e >= L::kKStages && !(ok = wait_bar(sh.k_empty[s], ((e / L::kKStages) - 1) & 1)))
            break;
          load_block(blk_lo + j, pid, sbase + L::kK + s * L::kTileBytes, bar(sh.k_full[s]), &tm_k,
                     &tm_kc, &tm_k8);
          issued_k = e + 1;
        } else {
          const int s = jg % L::kVStages;
          if (jg >= L::kVStages &&
              !(ok = wait_bar(sh.v_empty[s], ((jg / L::kVStages) - 1) & 1)))
            break;
          load_block(blk_lo + j, pid, sbase + L::kV + s * L::kTileBytes, bar(sh.v_full[s]), &tm_v,
                     &tm_vc, &tm_v8);
          issued_v = jg + 1;
        }
      }
      if (!ok) break;
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(sh.meta_empty[slot]));
      jbase += nb;
    }
    if (!ok && lane == 0) set_abort(sh, p.err);
    // Do not exit while a copy into this CTA's shared memory is in flight:
    // wait for the most recent phase of every barrier a copy may complete.
    for (int jg = max(0, issued_k - L::kKStages); jg < issued_k; ++jg)
      mbar_wait(bar(sh.k_full[jg % L::kKStages]), (jg / L::kKStages) & 1);
    for (int jg = max(0, issued_v - L::kVStages); jg < issued_v; ++jg)
      mbar_wait(bar(sh.v_full[jg % L::kVStages]), (jg / L::kVStages) & 1);
  } else if (warp == 1) {
    // ------------------------------------------------------ MMA issuer --
    // The whole warp runs this loop with warp-uniform values; one elected
    // lane issues each MMA / commit (see sm100.cuh).
    constexpr uint32_t idesc_qk = idesc_bf16_f32(kRows, kBlk, false);
    constexpr uint32_t idesc_pv = idesc_bf16_f32(kRows, D, true);
    // Shared-memory descriptors: a slot / stage / k-step offset only adds
    // (offset >> 4) to the start-address field (bits 0-13), which cannot
    // carry: every address stays below 256 KB.
    const uint64_t dk0 = smem_desc_sw128(sbase + L::kK, 16, 1024);
    // S[col] = Q (TMEM slot qs) K^T of global block jg: A from TMEM, 16
    // dimensions (8 columns) per MMA; B = K, K-major in shared memory
    // (one lane, elected once per group, issues the group's MMAs and commits)
    const bool issuer = elect_one();
    auto issue_qk = [&](int qs, int sk, uint32_t col) {
      const uint64_t kd = dk0 + ((sk * L::kTileBytes) >> 4);
      if (issuer) {
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = ((kk >> 2) * L::kChunkBytes + (kk & 3) * 32) >> 4;
          mma_ts_one(tmem + col, tmem + L::col_q(qs) + kk * 8, kd + off, idesc_qk, kk > 0);
        }
      }
      __syncwarp();
    };
    auto commit = [&](uint64_t &b) {
      if (issuer) mma_commit_one(bar(b));
      __syncwarp();
    };
    // O (+)= P V of global block jg, P in TMEM at column pcol: one
    // N = D MMA per 16 keys.  V is MN-major (D contiguous): 64-column swizzle
    // atoms kChunkBytes apart along N (leading byte offset), 8-key groups
    // 1024 bytes apart along K (stride byte offset).
    const uint64_t dv0 = smem_desc_sw128(sbase + L::kV, L::kChunkBytes, 1024);
    auto issue_pv = [&](int jg, bool first, uint32_t pcol) {
      const uint64_t vd = dv0 + (((jg % L::kVStages) * L::kTileBytes) >> 4);
      if (issuer) {
#pragma unroll
        for (int kk = 0; kk < kBlk / 16; ++kk)
          mma_ts_one(tmem + L::kColO, tmem + pcol + kk * 8, vd + ((kk * 16 * 128) >> 4), idesc_pv,
                     (!first || kk > 0) ? 1u : 0u);
      }
      __syncwarp();
    };
    auto wait = [&](uint64_t &b, int parity) {
      if (!wait_bar(b, parity)) return false;
      tc_fence_after();
      return true;
    };
    // The P V of a block is issued after the Q K^T of the next block (QK(b),
    // PV(b-1)), across unit boundaries too.
    struct Pending {
      int jg, unit;
      bool first, last;
    };
    Pending pend{0, 0, false, false};
    bool has_pend = false;
    // V of block x.jg and K of block jn (the next Q K^T) are tested while
    // the warp waits for P of block x.jg, so that their shared-memory round
    // trips overlap; only phases not yet complete are waited for again.
    // k_next: K of block jn has landed.
    // (jn: ring entry of the next K block, or -1 when the next entry is a Q)
    auto do_pv = [&](const Pending &x, int jn, bool &k_next) -> bool {
      const int s = x.jg & 1, sv = x.jg % L::kVStages;
      const int kb = jn >= 0 ? bar(sh.k_full[jn % L::kKStages]) : bar(sh.v_full[sv]);
      const int kp = jn >= 0 ? (jn / L::kKStages) & 1 : (x.jg / L::kVStages) & 1;
      uint32_t r = mbar_try_test2(bar(sh.p_full[s]), (x.jg >> 1) & 1, bar(sh.v_full[sv]),
                                  (x.jg / L::kVStages) & 1, kb, kp);
      r = __shfl_sync(0xffffffffu, r, 0);
      k_next = jn >= 0 && (r & 4u) != 0;
      if (!(r & 1u) && !wait_bar(sh.p_full[s], (x.jg >> 1) & 1)) return false;
      if (!(r & 2u) && !wait_bar(sh.v_full[sv], (x.jg / L::kVStages) & 1)) return false;
      tc_fence_after();
      // O last held unit x.unit - 1, whose epilogue must have read it
      if (x.first && x.unit >= 1 && !wait(sh.o_empty, (x.unit - 1) & 1)) return false;
      issue_pv(x.jg, x.first, L::col_s(s));
      commit(sh.pv_done);
      commit(sh.v_empty[sv]);
      if (x.last) commit(sh.o_full);
      return true;
    };
    int jbase = 0;
    bool ok = true, k_ready = false;
    for (int k = 0; ok; ++k) {
      const int slot = k & 1;
      if (!(ok = wait(sh.meta_full[slot], (k >> 1) & 1))) break;
      const bool valid = meta[slot].valid != 0;
      const int nb = meta[slot].n_blocks;
      __syncwarp();
      if (!valid) break;
      if (lane == 0) mbar_arrive(bar(sh.meta_empty[slot]));
      // the unit's Q: from its K-ring entry into TMEM slot qs (the copy runs
      // in order with the MMAs: unit k - 2's Q K^T are done with the slot)
      const int qs = k & 1, qe = jbase + k, sq = qe % L::kKStages;
      if (!(ok = wait(sh.k_full[sq], (qe / L::kKStages) & 1))) break;
      if (issuer) {
        const uint64_t qd = dk0 + ((sq * L::kTileBytes) >> 4);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk)
          tmem_cp_128x256b(tmem + L::col_q(qs) + kk * 8,
                           qd + (((kk >> 2) * L::kChunkBytes + (kk & 3) * 32) >> 4));
      }
      __syncwarp();
      commit(sh.k_empty[sq]);
      k_ready = false;
      for (int j = 0; j < nb; ++j) {
        const int jg = jbase + j, s = jg & 1, ke = jg + k + 1, sk = ke % L::kKStages;
        if (!k_ready && !(ok = wait(sh.k_full[sk], (ke / L::kKStages) & 1))) break;
        issue_qk(qs, sk, L::col_s(s));
        commit(sh.s_full[s]);
        commit(sh.k_empty[sk]);
        k_ready = false;
        if (has_pend && !(ok = do_pv(pend, j + 1 < nb ? ke + 1 : -1, k_ready))) break;
        pend = Pending{jg, k, j == 0, j == nb - 1};
        has_pend = true;
      }
      jbase += nb;
    }
    if (ok && has_pend) ok = do_pv(pend, -1, k_ready);
    if (!ok && lane == 0) set_abort(sh, p.err);
  } else {
    // --------------------------------------------------------- softmax --
    // Warpgroup half h owns key columns [64 h, 64 h + 64) of every block and
    // output columns [64 h, 64 h + 64).
    const int h = (warp - 2) >> 2;        // column half
    const int quad = warp & 3;            // TMEM lane quadrant this warp may access
    const int r_in = quad * 32 + lane;    // row within the tile
    const uint32_t t_lane = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    const float sl2 = p.scale_log2;
    // This thread's row of a unit: where it reads Q and writes the output,
    // and its visible keys (prefix below lim_p; own branch's private keys
    // j <= last, which start at packed page ps).
    struct Row {
      bool unit;  // false: no unit left
      bool valid;
      int g, split, nb, blk_lo, nP, lim_p, ps, last;
      size_t pair;
    };
    // Reads unit k's metadata (slot k & 1) and releases the slot (the unit's
    // Q reaches TMEM through the K ring and the MMA warp); false on timeout /
    // abort.
    auto begin_unit = [&](int k, Row &R) -> bool {
      const int slot = k & 1;
      if (!wait_bar(sh.meta_full[slot], (k >> 1) & 1)) return false;
      const UnitMeta &M = meta[slot];
      R.unit = M.valid != 0;
      if (R.unit) {
        R.g = M.g;
        R.split = M.split;
        R.nb = M.n_blocks;
        R.blk_lo = M.blk_lo;
        R.nP = M.nP;
        R.valid = r_in < M.nrows;
        const int token = M.tok0 + r_in / G;
        const int bl = R.valid ? token / m - M.b_lo : 0;
        R.lim_p = R.valid ? M.fork[bl] : 0;
        R.ps = R.valid ? M.page_start[bl] : 0;
        R.last = R.valid ? M.blen[bl] - m + (token - (M.b_lo + bl) * m) : -1;
        R.pair = static_cast<size_t>(token) * p.H_q + R.g * G + r_in % G;
      }
      __syncwarp();
      if (R.unit && lane == 0) mbar_arrive(bar(sh.meta_empty[slot]));
      return true;
    };
    const uint32_t o_col = L::kColO + h * (D / 2);
    int jbase = 0;
    Row cur{}, nxt{};
    bool ok = begin_unit(0, cur);
    for (int k = 0; ok && cur.unit; ++k) {
      float m_run = NEG_INF, l_half = 0.f;
      for (int j = 0; j < cur.nb; ++j) {
        const int jg = jbase + j;
        const int si = jg & 1;
        // warp-uniform outcome: the tcgen05.ld / st below are warp-collective
        if (!(ok = wait_bar(sh.s_full[si], (jg >> 1) & 1))) break;
        tc_fence_after();
        const int jb = cur.blk_lo + j;
        int lo, hi;
        if (jb < cur.nP) {
          lo = 0;
          hi = cur.lim_p - jb * kBlk;
        } else {
          const int off = (cur.ps - (jb - cur.nP) * kPagesPerBlock) * kPage;  // column of own key 0
          lo = max(0, off);
          hi = min(kBlk, off + cur.last + 1);
        }
        const int par = jg & 1;
        bool xok = true;
        auto xchg = [&](float mx) {
          sh.xmax[h][par][r_in] = mx;
          tc_fence_before();
          publish_seq(&sh.xseq[0][h][quad], jg + 1);
          xok = await_seq(&sh.xseq[0][h ^ 1][quad], jg + 1, sh);
          tc_fence_after();
          return fmaxf(mx, sh.xmax[h ^ 1][par][r_in]);
        };
        const float alpha =
            tc::softmax_half_tmem(t_lane + L::col_s(si), h, lo, hi, sl2, m_run, l_half, xchg);
        if (!(ok = __all_sync(0xffffffffu, xok))) break;
        // Before O may be rescaled, the P V MMA of block jg-1 must have
        // landed: a warp that rescales waits for it.  Warps skip the wait
        // when they do not rescale, yet the parity test stays exact: Q K^T
        // (jg) was issued after P V (jg-2), so the S commit awaited above
        // implies P V (jg-2) has completed, and P V (jg) needs this block's
        // P; the barrier is in one of two consecutive phases.
        const bool rescale = __any_sync(0xffffffffu, j > 0 && alpha != 1.f);
        if (rescale) {
          if (!(ok = wait_bar(sh.pv_done, (jg - 1) & 1))) break;
          tc_fence_after();
#pragma unroll
          for (int c = 0; c < D / 2; c += 32) {
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
      if (!ok) break;
      // the next unit's Q goes to TMEM before this unit's epilogue, so that
      // its first Q K^T MMAs run meanwhile
      if (!(ok = begin_unit(k + 1, nxt))) break;
      // ---------------------------------------------------- epilogue --
      // row sum over both halves
      sh.xsum[h][r_in] = l_half;
      publish_seq(&sh.xseq[1][h][quad], k + 1);
      if (!(ok = __all_sync(0xffffffffu, await_seq(&sh.xseq[1][h ^ 1][quad], k + 1, sh)))) break;
      const float l_run = l_half + sh.xsum[h ^ 1][r_in];
      if (!(ok = wait_bar(sh.o_full, k & 1))) break;
      tc_fence_after();
      const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
      const float lse = l_run > 0.f ? (m_run + __log2f(l_run)) * kLn2 : NEG_INF;
      const bool final_out = p.S_p == 1;
      const size_t slot_pair = static_cast<size_t>(cur.split) * p.rows_total * p.H_q + cur.pair;
#pragma unroll
      for (int c = 0; c < D / 2; c += 32) {
        uint32_t o[32];
        tmem_ld32(t_lane + o_col + c, o);
        tmem_ld_wait();
        if (!cur.valid) continue;
        const int dc = h * (D / 2) + c;  // output column
        // 32-byte stores: each fills a whole sector of its row
        if (final_out) {
          uint32_t w[16];
#pragma unroll
          for (int e = 0; e < 16; ++e)
            w[e] = pack_bf16x2(__uint_as_float(o[2 * e]) * inv, __uint_as_float(o[2 * e + 1]) * inv);
          __nv_bfloat16 *dst = p.out + cur.pair * D + dc;
          if (p.out_align32) {
            st_global_v8(dst, w);
            st_global_v8(dst + 16, w + 8);
          } else {
#pragma unroll
            for (int e = 0; e < 16; e += 4)
              reinterpret_cast<uint4 *>(dst)[e / 4] = make_uint4(w[e], w[e + 1], w[e + 2], w[e + 3]);
          }
        } else {
          float *dst = p.o_part + slot_pair * D + dc;
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * inv);
#pragma unroll
          for (int e = 0; e < 32; e += 8) st_global_v8(dst + e, o + e);
        }
      }
      if (cur.valid && h == 0) {
        if (final_out) {
          if (p.lse) p.lse[cur.pair] = lse;
        } else {
          p.l_part[slot_pair] = lse;
        }
      }
      // O may be overwritten by the next unit once every warp has read it
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(sh.o_empty));
      jbase += cur.nb;
      cur = nxt;
    }
    if (!ok && lane == 0) set_abort(sh, p.err);
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

template <int D>
cudaError_t launch_tc(const AttnParams &p, bool overlap, cudaStream_t s) {
  using L = TcLayout<D>;
  static_assert(L::kDynSmem + sizeof(TcShared) <= 227 * 1024, "shared memory");
  CUtensorMap tk, tv, tkc, tvc, tk8, tv8, tq;
  cudaError_t e = tc::make_prefix_maps(p, &tk, &tv);
  if (e == cudaSuccess) e = tc::make_q_map(p, &tq);
  if (e == cudaSuccess) e = tc::make_page_map(&tkc, p.k_cache, D, p.H_kv, p.num_pages);
  if (e == cudaSuccess) e = tc::make_page_map(&tvc, p.v_cache, D, p.H_kv, p.num_pages);
  const int run = std::min(kPagesPerBlock, p.num_pages);  // box never longer than the pool
  if (e == cudaSuccess) e = tc::make_page_map(&tk8, p.k_cache, D, p.H_kv, p.num_pages, run);
  if (e == cudaSuccess) e = tc::make_page_map(&tv8, p.v_cache, D, p.H_kv, p.num_pages, run);
  if (e != cudaSuccess) return e;
  static std::atomic<uint64_t> configured{0};
  int dev = 0;
  e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(configured.load(std::memory_order_acquire) & bit)) {
    e = cudaFuncSetAttribute(branch_attn_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
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
  const dim3 grid(static_cast<unsigned>(std::min(p.n_units, sms[dev & 63])), 1, 1);
  return launch_kernel(overlap, branch_attn_tc_kernel<D>, grid, dim3(kThreads), L::kDynSmem, s,
                       tk, tv, tkc, tvc, tk8, tv8, tq, p);
}

}  // namespace

cudaError_t launch_branch_attn_tc(const AttnParams &p, const Plan &plan, bool overlap,
                                  cudaStream_t s) {
  if (plan.tiles_max <= 0 || p.n_units <= 0) return cudaSuccess;
  return p.D == 64 ? launch_tc<64>(p, overlap, s) : launch_tc<128>(p, overlap, s);
}

}  // namespace hpd
