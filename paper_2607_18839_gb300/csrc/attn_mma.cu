// attn_mma.cu -- the two attention stages of the branch-decode step on
// warp-level bf16 tensor-core MMA (m16n8k16), producing split partials.
//
// Shared-prefix stage: for page d and KV head g, the query rows of ALL the
// page's branches that read KV head g are stacked (row r <-> token
// branch_cu[d]*m + r/G, query head g*G + r%G) and run against the page's
// prefix keys [0, P_d) as one dense problem, so each prefix K/V tile is read
// once per row tile instead of once per branch (the shared-prefix reuse of
// Sec. 3.3).  A per-branch fork-position prefix length masks each row's tail.
//
// Private-suffix stage: for branch b and KV head g, the m*G rows of the
// branch read only that branch's paged keys, with the causal rule
// j <= L_b - m + i among the m P-MTP queries (Sec. 3.3, Sec. 3.4).
//
// Both stages split their key range into chunks and write, per chunk, the
// normalised partial output O_s (fp32) and its log-sum-exp lse_s (natural
// log; -inf when the chunk holds no visible key).  The suffix stage combines
// them: for each branch, the last of its suffix CTAs to finish merges every
// slot of the branch's rows by log-sum-exp and writes out / lse.
#include <atomic>

#include "common.cuh"

namespace hpd {
namespace {

constexpr int kThreads = 128;  // 4 warps
constexpr int kBN = 64;        // keys per shared-memory block
constexpr int kMaxSlots = 17;  // prefix splits + suffix splits + own partial

// Byte offset of 16-byte chunk `c` of row `r` in a row-major tile of D bf16
// columns; chunks are XOR-swizzled by the row so ldmatrix is conflict-free.
template <int D>
__device__ __forceinline__ uint32_t tile_off(int r, int c) {
  return static_cast<uint32_t>(r * D * 2 + ((c ^ (r & 7)) << 4));
}

template <int D, int WR, bool PREFIX>
__global__ void __launch_bounds__(kThreads) attn_stage_kernel(const AttnParams p) {
  constexpr int WK = 4 / WR;      // warps along keys
  constexpr int TILE_M = 16 * WR; // query rows per CTA
  constexpr int NK = kBN / WK;    // keys per warp per block
  constexpr int NT = NK / 8;      // S n-tiles per warp
  constexpr int DC = D / 8;       // 16-byte chunks per row
  constexpr int KD = D / 16;      // k-steps over the head dim
  constexpr int DT = D / 8;       // O n-tiles
  static_assert(NT % 2 == 0, "key tiles are loaded in pairs");

  extern __shared__ __align__(128) uint8_t smem[];
  uint8_t *sQ = smem;
  uint8_t *sK = sQ + TILE_M * D * 2;
  uint8_t *sV = sK + 2 * kBN * D * 2;
  __shared__ int s_info[4];

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int rg = warp % WR, kg = warp / WR;
  const int G = p.G, m = p.m;
  const float NEG_INF = -__int_as_float(0x7f800000);

  // ------------------------------------------------------ work decode --
  int g, slot, r0, nrows, tokbase, k_begin, k_end;
  int pc0 = 0, bidx = 0, L = 0, P_d = 0, doc = 0;
  if constexpr (PREFIX) {
    g = blockIdx.y;
    const int split = blockIdx.z;
    slot = split;
    const int tile = blockIdx.x;
    if (tid == 0) s_info[0] = -1;
    __syncthreads();
    if (warp == 0) {
      // Find the page owning this row tile: page d has ceil(R_d / TILE_M)
      // tiles, R_d = (#branches of d) * m * G.
      int base = 0;
      for (int d0 = 0; d0 < p.n_docs; d0 += 32) {
        const int d = d0 + lane;
        int tiles = 0, b0 = 0, b1 = 0;
        if (d < p.n_docs) {
          b0 = min(max(p.branch_cu[d], 0), p.B);
          b1 = min(max(p.branch_cu[d + 1], 0), p.B);
          if (b1 < b0) { flag_error(p.err, HPD_DEVERR_BRANCH_CU); b1 = b0; }
          tiles = ceil_div_i((b1 - b0) * m * G, TILE_M);
        }
        int incl = tiles;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int v = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += v;
        }
        const int excl = incl - tiles;
        if (tiles > 0 && tile >= base + excl && tile < base + incl) {
          s_info[0] = d;
          s_info[1] = tile - base - excl;
          s_info[2] = b0;
          s_info[3] = b1;
        }
        base += __shfl_sync(0xffffffffu, incl, 31);
        if (base > tile) break;
      }
    }
    __syncthreads();
    const int d = s_info[0];
    if (d < 0) return;  // grid is an upper bound of the tile count
    const int lt = s_info[1], b0 = s_info[2], b1 = s_info[3];
    bool bad;
    page_prefix(p, d, pc0, P_d, bad);
    if (bad) flag_error(p.err, HPD_DEVERR_PREFIX_CU);
    doc = d;
    const int R_d = (b1 - b0) * m * G;
    r0 = lt * TILE_M;
    nrows = min(TILE_M, R_d - r0);
    tokbase = b0 * m;
    const int chunk = ceil_div_i(ceil_div_i(max(P_d, 1), p.S_p), kBN) * kBN;
    k_begin = split * chunk;
    k_end = min(P_d, k_begin + chunk);
  } else {
    bidx = blockIdx.x;
    const int rt_s = ceil_div_i(m * G, TILE_M);
    g = blockIdx.y / rt_s;
    const int rt = blockIdx.y % rt_s;
    const int split = blockIdx.z;
    slot = p.S_p + split;
    r0 = rt * TILE_M;
    nrows = min(TILE_M, m * G - r0);
    tokbase = bidx * m;
    int Lraw = p.branch_len[bidx];
    const int Lcap = p.max_pages * kPage;
    if (Lraw < 0 || Lraw > Lcap) {
      if (tid == 0) flag_error(p.err, HPD_DEVERR_BRANCH_LEN);
      Lraw = min(max(Lraw, 0), Lcap);
    }
    L = Lraw;
    const int chunk = ceil_div_i(ceil_div_i(max(L, 1), p.S_s), kBN) * kBN;
    k_begin = split * chunk;
    k_end = min(L, k_begin + chunk);
    // the last private key any row of this tile may see
    const int i_max = (r0 + nrows - 1) / G;
    k_end = min(k_end, L - m + i_max + 1);
  }

  // Exclusive key limits of this thread's two rows (tile-local ra, rb).
  const int ra = rg * 16 + (lane >> 2), rb = ra + 8;
  auto row_limit = [&](int r) -> int {
    if (r >= nrows) return k_begin;  // padding row: sees nothing
    int lim = k_end;
    if constexpr (PREFIX) {
      if (p.branch_prefix_len) {
        const int b = (tokbase + (r0 + r) / G) / m;
        int f = p.branch_prefix_len[b];
        if (f < 0 || f > P_d) { flag_error(p.err, HPD_DEVERR_FORK_LEN); f = min(max(f, 0), P_d); }
        lim = min(lim, f);
      }
    } else {
      const int i = (r0 + r) / G;
      lim = min(lim, L - m + i + 1);
    }
    return lim;
  };
  const int lim_a = row_limit(ra), lim_b = row_limit(rb);

  // The furthest key any row needs: shrink the loop for short fork prefixes.
  if constexpr (PREFIX) {
    if (p.branch_prefix_len) {
      __shared__ int s_kmax;
      if (tid == 0) s_kmax = k_begin;
      __syncthreads();
      if ((lane & 3) == 0) {
        atomicMax(&s_kmax, lim_a);
        atomicMax(&s_kmax, lim_b);
      }
      __syncthreads();
      k_end = min(k_end, s_kmax);
    }
  }

  const size_t HD = static_cast<size_t>(p.H_q) * D;
  auto out_index = [&](int r) -> size_t {  // (slot, token, head) of tile row r
    const int token = tokbase + (r0 + r) / G;
    const int head = g * G + (r0 + r) % G;
    return (static_cast<size_t>(slot) * p.rows_total + token) * p.H_q + head;
  };

  if (nrows <= 0) return;
  const bool empty = k_end <= k_begin;
  if (PREFIX && empty) {
    for (int r = tid; r < nrows; r += kThreads) p.l_part[out_index(r)] = NEG_INF;
    return;
  }

  // --------------------------------------------------------- loaders --
  const bool pool = !PREFIX || p.prefix_page_table;
  const __nv_bfloat16 *Kbase = pool ? p.k_cache : p.prefix_k;
  const __nv_bfloat16 *Vbase = pool ? p.v_cache : p.prefix_v;
  auto key_row = [&](int j) -> size_t {  // element offset of key j's head-g vector
    if constexpr (PREFIX) {
      if (p.prefix_page_table)  // paged prefix: slot j % 16 of a pool page
        return ((static_cast<size_t>(prefix_page(p, doc, j / kPage)) * kPage + (j % kPage)) *
                    p.H_kv + g) * D;
      return (static_cast<size_t>(pc0 + j) * p.H_kv + g) * D;
    } else {
      int page = p.page_table[static_cast<size_t>(bidx) * p.max_pages + j / kPage];
      if (page < 0 || page >= p.num_pages) { flag_error(p.err, HPD_DEVERR_PAGE_ID); page = 0; }
      return ((static_cast<size_t>(page) * kPage + (j % kPage)) * p.H_kv + g) * D;
    }
  };
  auto load_kv = [&](int kb0, int buf) {
    const uint32_t dk = smem_u32(sK + buf * kBN * D * 2);
    const uint32_t dv = smem_u32(sV + buf * kBN * D * 2);
#pragma unroll
    for (int it = 0; it < (kBN * DC) / kThreads; ++it) {
      const int idx = tid + it * kThreads;
      const int row = idx / DC, c = idx % DC;
      const int j = kb0 + row;
      const bool ok = j < k_end;
      const size_t off = ok ? key_row(j) + c * 8 : 0;
      cp_async16(dk + tile_off<D>(row, c), Kbase + off, ok ? 16 : 0);
      cp_async16(dv + tile_off<D>(row, c), Vbase + off, ok ? 16 : 0);
    }
  };
  if (!empty) {
    const uint32_t dq = smem_u32(sQ);
    for (int idx = tid; idx < TILE_M * DC; idx += kThreads) {
      const int row = idx / DC, c = idx % DC;
      const bool ok = row < nrows;
      size_t off = 0;
      if (ok) {
        const int token = tokbase + (r0 + row) / G;
        const int head = g * G + (r0 + row) % G;
        off = static_cast<size_t>(token) * HD + static_cast<size_t>(head) * D + c * 8;
      }
      cp_async16(dq + tile_off<D>(row, c), p.q + off, ok ? 16 : 0);
    }
    load_kv(k_begin, 0);
    cp_async_commit();
  }

  // ---------------------------------------------------------- main loop --
  uint32_t qf[KD][4];
  float o[DT][4];
#pragma unroll
  for (int i = 0; i < DT; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m_a = NEG_INF, m_b = NEG_INF, l_a = 0.f, l_b = 0.f;
  const float sl2 = p.scale_log2;

  const int n_blocks = empty ? 0 : ceil_div_i(k_end - k_begin, kBN);
  for (int blk = 0; blk < n_blocks; ++blk) {
    const int kb0 = k_begin + blk * kBN;
    if (blk + 1 < n_blocks) {
      load_kv(kb0 + kBN, (blk + 1) & 1);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    if (blk == 0) {
      const uint32_t q0 = smem_u32(sQ);
#pragma unroll
      for (int kk = 0; kk < KD; ++kk) {
        const int row = rg * 16 + (lane & 15);
        const int c = kk * 2 + (lane >> 4);
        ldmatrix_x4(q0 + tile_off<D>(row, c), qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3]);
      }
    }
    const uint32_t kbuf = smem_u32(sK + (blk & 1) * kBN * D * 2);
    const uint32_t vbuf = smem_u32(sV + (blk & 1) * kBN * D * 2);
    const int kw = kg * NK;  // first key of this warp inside the block

    // S = Q K^T for 16 rows x NK keys
    float s[NT][4];
#pragma unroll
    for (int i = 0; i < NT; ++i) s[i][0] = s[i][1] = s[i][2] = s[i][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < KD; ++kk) {
#pragma unroll
      for (int nt = 0; nt < NT; nt += 2) {
        uint32_t b0, b1, b2, b3;
        const int key = kw + nt * 8 + ((lane >> 4) << 3) + (lane & 7);
        const int c = kk * 2 + ((lane >> 3) & 1);
        ldmatrix_x4(kbuf + tile_off<D>(key, c), b0, b1, b2, b3);
        mma_bf16_16816(s[nt], qf[kk], b0, b1);
        mma_bf16_16816(s[nt + 1], qf[kk], b2, b3);
      }
    }

    // mask + online softmax (base 2)
    float mx_a = NEG_INF, mx_b = NEG_INF;
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int j = kb0 + kw + nt * 8 + (lane & 3) * 2 + e;
        const float va = j < lim_a ? s[nt][e] * sl2 : NEG_INF;
        const float vb = j < lim_b ? s[nt][2 + e] * sl2 : NEG_INF;
        s[nt][e] = va;
        s[nt][2 + e] = vb;
        mx_a = fmaxf(mx_a, va);
        mx_b = fmaxf(mx_b, vb);
      }
    }
    mx_a = fmaxf(mx_a, __shfl_xor_sync(0xffffffffu, mx_a, 1));
    mx_a = fmaxf(mx_a, __shfl_xor_sync(0xffffffffu, mx_a, 2));
    mx_b = fmaxf(mx_b, __shfl_xor_sync(0xffffffffu, mx_b, 1));
    mx_b = fmaxf(mx_b, __shfl_xor_sync(0xffffffffu, mx_b, 2));
    const float mn_a = fmaxf(m_a, mx_a), mn_b = fmaxf(m_b, mx_b);
    const float base_a = mn_a == NEG_INF ? 0.f : mn_a;
    const float base_b = mn_b == NEG_INF ? 0.f : mn_b;
    const float alpha_a = fast_exp2(m_a - base_a), alpha_b = fast_exp2(m_b - base_b);
    m_a = mn_a;
    m_b = mn_b;
    float sum_a = 0.f, sum_b = 0.f;
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      s[nt][0] = fast_exp2(s[nt][0] - base_a);
      s[nt][1] = fast_exp2(s[nt][1] - base_a);
      s[nt][2] = fast_exp2(s[nt][2] - base_b);
      s[nt][3] = fast_exp2(s[nt][3] - base_b);
      sum_a += s[nt][0] + s[nt][1];
      sum_b += s[nt][2] + s[nt][3];
    }
    l_a = l_a * alpha_a + sum_a;
    l_b = l_b * alpha_b + sum_b;
#pragma unroll
    for (int dt = 0; dt < DT; ++dt) {
      o[dt][0] *= alpha_a;
      o[dt][1] *= alpha_a;
      o[dt][2] *= alpha_b;
      o[dt][3] *= alpha_b;
    }

    // O += P V
#pragma unroll
    for (int kc = 0; kc < NT / 2; ++kc) {
      uint32_t a[4];
      a[0] = pack_bf16x2(s[2 * kc][0], s[2 * kc][1]);
      a[1] = pack_bf16x2(s[2 * kc][2], s[2 * kc][3]);
      a[2] = pack_bf16x2(s[2 * kc + 1][0], s[2 * kc + 1][1]);
      a[3] = pack_bf16x2(s[2 * kc + 1][2], s[2 * kc + 1][3]);
#pragma unroll
      for (int dt = 0; dt < DT; dt += 2) {
        uint32_t b0, b1, b2, b3;
        const int key = kw + kc * 16 + (((lane >> 3) & 1) << 3) + (lane & 7);
        const int c = dt + (lane >> 4);
        ldmatrix_x4_trans(vbuf + tile_off<D>(key, c), b0, b1, b2, b3);
        mma_bf16_16816(o[dt], a, b0, b1);
        mma_bf16_16816(o[dt + 1], a, b2, b3);
      }
    }
    __syncthreads();  // the next iteration's prefetch overwrites this buffer
  }

  l_a += __shfl_xor_sync(0xffffffffu, l_a, 1);
  l_a += __shfl_xor_sync(0xffffffffu, l_a, 2);
  l_b += __shfl_xor_sync(0xffffffffu, l_b, 1);
  l_b += __shfl_xor_sync(0xffffffffu, l_b, 2);

  // ------------------------------------------------------------ epilogue --
  // Normalised partial of this CTA's rows: prefix stage -> its workspace
  // slot; suffix stage -> shared memory, then merged with the other slots.
  float *sm_m = reinterpret_cast<float *>(sK);  // [WK][TILE_M]
  float *sm_l = sm_m + WK * TILE_M;             // [WK][TILE_M]
  float *sm_M = sm_l + WK * TILE_M;             // [TILE_M]
  float *sm_L = sm_M + TILE_M;                  // [TILE_M]
  float *sm_o = sm_L + TILE_M;                  // [WK][TILE_M][D]; slice 0 = own partial
  float *sm_lse = sm_o + WK * TILE_M * D;       // [TILE_M] own partial lse
  float *sm_inv = sm_lse + TILE_M;              // [TILE_M]
  float *sm_w = sm_inv + TILE_M;                // [TILE_M][kMaxSlots]
  if constexpr (WK == 1) {
    const float inv_a = l_a > 0.f ? 1.f / l_a : 0.f;
    const float inv_b = l_b > 0.f ? 1.f / l_b : 0.f;
    const float lse_a = l_a > 0.f ? (m_a + __log2f(l_a)) * kLn2 : NEG_INF;
    const float lse_b = l_b > 0.f ? (m_b + __log2f(l_b)) * kLn2 : NEG_INF;
    if constexpr (PREFIX) {
      if (ra < nrows) {
        float *dst = p.o_part + out_index(ra) * D;
#pragma unroll
        for (int dt = 0; dt < DT; ++dt)
          *reinterpret_cast<float2 *>(dst + dt * 8 + (lane & 3) * 2) =
              make_float2(o[dt][0] * inv_a, o[dt][1] * inv_a);
        if ((lane & 3) == 0) p.l_part[out_index(ra)] = lse_a;
      }
      if (rb < nrows) {
        float *dst = p.o_part + out_index(rb) * D;
#pragma unroll
        for (int dt = 0; dt < DT; ++dt)
          *reinterpret_cast<float2 *>(dst + dt * 8 + (lane & 3) * 2) =
              make_float2(o[dt][2] * inv_b, o[dt][3] * inv_b);
        if ((lane & 3) == 0) p.l_part[out_index(rb)] = lse_b;
      }
      return;
    } else {
#pragma unroll
      for (int dt = 0; dt < DT; ++dt) {
        const int d = dt * 8 + (lane & 3) * 2;
        *reinterpret_cast<float2 *>(sm_o + ra * D + d) = make_float2(o[dt][0] * inv_a, o[dt][1] * inv_a);
        *reinterpret_cast<float2 *>(sm_o + rb * D + d) = make_float2(o[dt][2] * inv_b, o[dt][3] * inv_b);
      }
      if ((lane & 3) == 0) {
        sm_lse[ra] = lse_a;
        sm_lse[rb] = lse_b;
      }
    }
  } else {
    // Combine the WK key groups of each row (the K/V buffers are free after
    // the loop's final barrier).
    if ((lane & 3) == 0) {
      sm_m[kg * TILE_M + ra] = m_a;
      sm_l[kg * TILE_M + ra] = l_a;
      sm_m[kg * TILE_M + rb] = m_b;
      sm_l[kg * TILE_M + rb] = l_b;
    }
    __syncthreads();
    if (tid < TILE_M) {
      float M = NEG_INF;
      for (int k = 0; k < WK; ++k) M = fmaxf(M, sm_m[k * TILE_M + tid]);
      const float base = M == NEG_INF ? 0.f : M;
      float Ls = 0.f;
      for (int k = 0; k < WK; ++k) Ls += sm_l[k * TILE_M + tid] * fast_exp2(sm_m[k * TILE_M + tid] - base);
      sm_M[tid] = M;
      sm_L[tid] = Ls;
    }
    __syncthreads();
    {
      const float Ma = sm_M[ra], Mb = sm_M[rb];
      const float fa = fast_exp2(m_a - (Ma == NEG_INF ? 0.f : Ma));
      const float fb = fast_exp2(m_b - (Mb == NEG_INF ? 0.f : Mb));
#pragma unroll
      for (int dt = 0; dt < DT; ++dt) {
        const int d = dt * 8 + (lane & 3) * 2;
        *reinterpret_cast<float2 *>(sm_o + (kg * TILE_M + ra) * D + d) =
            make_float2(o[dt][0] * fa, o[dt][1] * fa);
        *reinterpret_cast<float2 *>(sm_o + (kg * TILE_M + rb) * D + d) =
            make_float2(o[dt][2] * fb, o[dt][3] * fb);
      }
    }
    __syncthreads();
    // sum the key groups into slice 0 (each element read and written by one thread)
    for (int idx = tid; idx < TILE_M * (D / 4); idx += kThreads) {
      const int r = idx / (D / 4), d = (idx % (D / 4)) * 4;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int k = 0; k < WK; ++k) {
        const float4 v = *reinterpret_cast<const float4 *>(sm_o + (k * TILE_M + r) * D + d);
        acc.x += v.x; acc.y += v.y; acc.z += v.z; acc.w += v.w;
      }
      const float Ls = sm_L[r];
      const float inv = Ls > 0.f ? 1.f / Ls : 0.f;
      acc.x *= inv; acc.y *= inv; acc.z *= inv; acc.w *= inv;
      if constexpr (PREFIX) {
        if (r < nrows) *reinterpret_cast<float4 *>(p.o_part + out_index(r) * D + d) = acc;
      } else {
        *reinterpret_cast<float4 *>(sm_o + r * D + d) = acc;
      }
    }
    for (int r = tid; r < TILE_M; r += kThreads) {
      const float Ls = sm_L[r];
      const float lse_r = Ls > 0.f ? (sm_M[r] + __log2f(Ls)) * kLn2 : NEG_INF;
      if constexpr (PREFIX) {
        if (r < nrows) p.l_part[out_index(r)] = lse_r;
      } else {
        sm_lse[r] = lse_r;
      }
    }
    if constexpr (PREFIX) return;
  }

  if constexpr (!PREFIX) {
    // ---- LSE merge of this branch's rows:
    //   out = sum_s e^{lse_s - M} O_s / sum_s e^{lse_s - M},
    //   lse = M + ln sum_s e^{lse_s - M},  M = max_s lse_s,
    // over the prefix splits and the suffix splits of the branch.  The union
    // of their key ranges is exactly the branch's visible key set (Sec. 3.3),
    // so this equals one softmax over all of it.  A partial whose range held
    // no visible key has lse_s = -inf and weight 0.
    __shared__ int s_last;
    bool own_in_smem = true;
    if (p.S_s > 1) {
      // Several CTAs hold this branch's suffix: publish this CTA's partial;
      // the last CTA to arrive merges them all (no CTA ever waits).
      __syncthreads();
      for (int idx = tid; idx < nrows * (D / 4); idx += kThreads) {
        const int r = idx / (D / 4), d = (idx % (D / 4)) * 4;
        *reinterpret_cast<float4 *>(p.o_part + out_index(r) * D + d) =
            *reinterpret_cast<const float4 *>(sm_o + r * D + d);
      }
      for (int r = tid; r < nrows; r += kThreads) p.l_part[out_index(r)] = sm_lse[r];
      __threadfence();
      __syncthreads();
      int *ctr = p.counters + (static_cast<size_t>(bidx) * p.H_kv + g) * ceil_div_i(m * G, TILE_M) +
                 r0 / TILE_M;
      if (tid == 0) s_last = atomicAdd(ctr, 1) == p.S_s - 1;
      __syncthreads();
      if (!s_last) return;
      __threadfence();
      if (tid == 0) atomicExch(ctr, 0);
      own_in_smem = false;
    }
    __syncthreads();
    const int n_glob = own_in_smem ? p.S_p : p.S_p + p.S_s;  // partials read from the workspace
    auto slot_index = [&](int s, int r) -> size_t {
      const int token = tokbase + (r0 + r) / G;
      const int head = g * G + (r0 + r) % G;
      return (static_cast<size_t>(s) * p.rows_total + token) * p.H_q + head;
    };
    // weights: one row per thread, all of the row's lse loads in flight
    static_assert(16 * WR <= kThreads, "one thread per row");
    if (tid < nrows) {
      const int r = tid;
      float ls[kMaxSlots];
#pragma unroll
      for (int s = 0; s < kMaxSlots; ++s)
        ls[s] = s < n_glob ? p.l_part[slot_index(s, r)] : NEG_INF;
      float M = own_in_smem ? sm_lse[r] : NEG_INF;
#pragma unroll
      for (int s = 0; s < kMaxSlots; ++s) M = fmaxf(M, ls[s]);
      float wsum = 0.f;
#pragma unroll
      for (int s = 0; s < kMaxSlots; ++s) {
        const float w = ls[s] == NEG_INF ? 0.f : __expf(ls[s] - M);
        if (s < n_glob) sm_w[r * kMaxSlots + s] = w;
        wsum += w;
      }
      const float w_own = own_in_smem && sm_lse[r] != NEG_INF ? __expf(sm_lse[r] - M) : 0.f;
      sm_w[r * kMaxSlots + n_glob] = w_own;
      wsum += w_own;
      sm_inv[r] = wsum > 0.f ? 1.f / wsum : 0.f;
      if (p.lse) p.lse[slot_index(0, r)] = M == NEG_INF ? NEG_INF : M + logf(wsum);
    }
    __syncthreads();
    // outputs: each thread owns up to kElems (row, 4-column) elements and, per
    // partial, issues all of their loads before accumulating
    constexpr int kElems = (16 * WR * (D / 4) + kThreads - 1) / kThreads;
    const int total = nrows * (D / 4);
    float4 acc[kElems];
#pragma unroll
    for (int u = 0; u < kElems; ++u) {
      acc[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      const int idx = tid + u * kThreads;
      if (own_in_smem && idx < total) {
        const int r = idx / (D / 4), d = (idx % (D / 4)) * 4;
        const float w = sm_w[r * kMaxSlots + n_glob];
        const float4 v = *reinterpret_cast<const float4 *>(sm_o + r * D + d);
        acc[u] = make_float4(w * v.x, w * v.y, w * v.z, w * v.w);
      }
    }
    for (int s = 0; s < n_glob; ++s) {
      float4 v[kElems];
      float w[kElems];
#pragma unroll
      for (int u = 0; u < kElems; ++u) {
        const int idx = tid + u * kThreads;
        const int r = idx / (D / 4), d = (idx % (D / 4)) * 4;
        w[u] = idx < total ? sm_w[r * kMaxSlots + s] : 0.f;
        v[u] = w[u] != 0.f
                   ? *reinterpret_cast<const float4 *>(p.o_part + slot_index(s, r) * D + d)
                   : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int u = 0; u < kElems; ++u) {
        acc[u].x += w[u] * v[u].x;
        acc[u].y += w[u] * v[u].y;
        acc[u].z += w[u] * v[u].z;
        acc[u].w += w[u] * v[u].w;
      }
    }
#pragma unroll
    for (int u = 0; u < kElems; ++u) {
      const int idx = tid + u * kThreads;
      if (idx < total) {
        const int r = idx / (D / 4), d = (idx % (D / 4)) * 4;
        const float inv = sm_inv[r];
        uint2 packed;
        packed.x = pack_bf16x2(acc[u].x * inv, acc[u].y * inv);
        packed.y = pack_bf16x2(acc[u].z * inv, acc[u].w * inv);
        *reinterpret_cast<uint2 *>(p.out + slot_index(0, r) * D + d) = packed;
      }
    }
  }
}

template <int D, int WR, bool PREFIX>
size_t stage_smem() {
  return static_cast<size_t>(16 * WR) * D * 2 + 2ull * 2 * kBN * D * 2;
}
// The epilogue scratch (per-row stats, own partial, merge weights) lives in
// the K/V buffers.
template <int D, int WR>
constexpr size_t epilogue_floats() {
  return (2 * (4 / WR) + 4) * (16 * WR) + (4 / WR) * (16 * WR) * D + (16 * WR) * kMaxSlots;
}
static_assert(epilogue_floats<128, 1>() * 4 <= 4 * kBN * 128 * 2, "epilogue scratch");
static_assert(epilogue_floats<128, 4>() * 4 <= 4 * kBN * 128 * 2, "epilogue scratch");
static_assert(epilogue_floats<64, 1>() * 4 <= 4 * kBN * 64 * 2, "epilogue scratch");
static_assert(epilogue_floats<64, 4>() * 4 <= 4 * kBN * 64 * 2, "epilogue scratch");

template <int D, int WR, bool PREFIX>
cudaError_t launch_stage(const AttnParams &p, dim3 grid, cudaStream_t s) {
  const size_t smem = stage_smem<D, WR, PREFIX>();
  // The shared-memory opt-in is a per-device function attribute: set it once
  // per device (outside any stream capture, on the first call).
  static std::atomic<uint64_t> configured{0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(configured.load(std::memory_order_acquire) & bit)) {
    e = cudaFuncSetAttribute(attn_stage_kernel<D, WR, PREFIX>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    configured.fetch_or(bit, std::memory_order_acq_rel);
  }
  attn_stage_kernel<D, WR, PREFIX><<<grid, kThreads, smem, s>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_prefix_stage(const AttnParams &p, const Plan &plan, cudaStream_t s) {
  if (plan.tiles_max <= 0) return cudaSuccess;
  const dim3 grid(plan.tiles_max, p.H_kv, plan.S_p);
  return p.D == 64 ? launch_stage<64, 4, true>(p, grid, s) : launch_stage<128, 4, true>(p, grid, s);
}

cudaError_t launch_suffix_stage(const AttnParams &p, const Plan &plan, cudaStream_t s) {
  const dim3 grid(p.B, p.H_kv * plan.rt_s, plan.S_s);
  if (p.D == 64) {
    if (plan.wr_s == 1) return launch_stage<64, 1, false>(p, grid, s);
    if (plan.wr_s == 2) return launch_stage<64, 2, false>(p, grid, s);
    return launch_stage<64, 4, false>(p, grid, s);
  }
  if (plan.wr_s == 1) return launch_stage<128, 1, false>(p, grid, s);
  if (plan.wr_s == 2) return launch_stage<128, 2, false>(p, grid, s);
  return launch_stage<128, 4, false>(p, grid, s);
}

}  // namespace hpd
