/*
 * hpd_oracle.c -- plain fp64 CPU oracle for one branch-decode step of
 * Hierarchical Parallel Decoding (HPD-Parsing).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the correctness reference the CUDA
 * library is checked against.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg may load it; the product path never does.  It
 * shares no code, header, table or helper with the CUDA library.
 *
 * What it computes (direct loops, no blocking, no fusion, no reordering):
 *
 *  1. Branch attention (Sec. 3.3, "Dynamic Branch Forking and Efficient
 *     Context Isolation"): a content branch attends to the shared visual
 *     context plus the layout prefix available at its fork position, and to
 *     its own incremental content KV cache -- never to other branches.
 *     Each branch carries m P-MTP query tokens (Sec. 3.4, "Integration with
 *     P-MTP"), which are causal among themselves.  For branch b of page d,
 *     query i in [0, m), query head h, KV head g = h / (H_q / H_kv)
 *     (grouped-query attention, Sec. 3.2 "LLM Decoder"), the visible keys are
 *        prefix keys   j in [0, P_b)                 (P_b = P_d unless a
 *                                                     per-branch fork length
 *                                                     is given)
 *        private keys  j in [0, L_b - m + i]         (L_b includes the m
 *                                                     tokens of this step)
 *     Private key j lives in physical page page_table[b][j / 16], slot j % 16.
 *     The prefix is either contiguous (page d's keys are rows
 *     [prefix_cu[d], prefix_cu[d+1]) of prefix_k / prefix_v) or paged in the
 *     same pool as the private keys, shared by every branch of the page
 *     without a copy (Algorithm 1's fork shares the parent's KV pages):
 *     prefix key j of page d is slot j % 16 of physical page
 *     prefix_page_table[d][j / 16].
 *     With s_j = scale * <q, k_j> over the visible set K:
 *        M   = max_j s_j
 *        out = sum_j exp(s_j - M) v_j / sum_j exp(s_j - M)
 *        lse = M + ln sum_j exp(s_j - M)            (natural log)
 *     An empty visible set gives out = 0 and lse = -inf.
 *
 *  2. Greedy P-MTP acceptance (Sec. 3.4; Algorithm 1, the verification step):
 *        t*_{b,j} = argmax_v logits[b][j][v], the lowest index on ties; NaN
 *                   entries never win (an all-NaN row gives index 0)
 *        n_acc_b  = largest k <= m with drafts[b][i] == t*_{b,i} for all i < k
 *
 * All floating-point inputs are bfloat16 bit patterns (uint16), widened
 * exactly to double.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORACLE_PAGE 16

static double bf16_to_double(uint16_t bits) {
  uint32_t w = ((uint32_t)bits) << 16;
  float f;
  memcpy(&f, &w, sizeof f);
  return (double)f;
}

/* Number of threads an OpenMP region will use (1 without OpenMP). */
int oracle_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

/*
 * Branch attention, item 1 above.
 *
 * q        [B*m][H_q][D]            row b*m + i (branch-major)
 * prefix_k [sum_d P_d][H_kv][D]      page d's prefix is tokens
 * prefix_v                           [prefix_cu[d], prefix_cu[d+1])
 * branch_cu [n_docs+1]               branches of page d are
 *                                    [branch_cu[d], branch_cu[d+1])
 * branch_prefix_len [B] or NULL      fork-position prefix length (<= P_d)
 * k_cache, v_cache [num_pages][16][H_kv][D]
 * page_table [B][max_pages]
 * branch_len [B]                     L_b, private entries incl. this step's m
 * branch_sel [n_sel] or NULL         compute only these branches (NULL: all)
 * prefix_page_table [n_docs][max_prefix_pages] or NULL
 *                                    paged prefix in k_cache / v_cache;
 *                                    prefix_k / prefix_v are then unused
 * out [B*m][H_q][D], lse [B*m][H_q]  written only for the computed branches
 *
 * Returns 0, or -1 on an index that falls outside its buffer.
 */
int oracle_branch_attn(const uint16_t *q, const uint16_t *prefix_k,
                       const uint16_t *prefix_v, const int32_t *prefix_cu,
                       const int32_t *branch_cu,
                       const int32_t *branch_prefix_len,
                       const uint16_t *k_cache, const uint16_t *v_cache,
                       const int32_t *page_table, const int32_t *branch_len,
                       int n_docs, int B, int m, int H_q, int H_kv, int D,
                       int num_pages, int max_pages, double scale,
                       const int32_t *branch_sel, int n_sel, int n_threads,
                       double *out, double *lse, const int32_t *prefix_page_table,
                       int max_prefix_pages) {
  if (H_kv <= 0 || H_q % H_kv != 0) return -1;
  const int G = H_q / H_kv;
  const int n_branches = branch_sel ? n_sel : B;
  int bad = 0;
#ifdef _OPENMP
  if (n_threads > 0) omp_set_num_threads(n_threads);
#else
  (void)n_threads;
#endif

  /* One task per (selected branch, query head); each handles the m queries. */
#pragma omp parallel for schedule(dynamic, 1) reduction(| : bad)
  for (long task = 0; task < (long)n_branches * H_q; ++task) {
    const int b = branch_sel ? branch_sel[task / H_q] : (int)(task / H_q);
    const int h = (int)(task % H_q);
    const int g = h / G;

    /* page d that owns branch b */
    int d = -1;
    for (int dd = 0; dd < n_docs; ++dd)
      if (b >= branch_cu[dd] && b < branch_cu[dd + 1]) d = dd;
    if (d < 0) { bad = 1; continue; }
    const int P_d = prefix_cu[d + 1] - prefix_cu[d];
    int P_b = branch_prefix_len ? branch_prefix_len[b] : P_d;
    if (P_b < 0 || P_b > P_d) { bad = 1; continue; }
    if (prefix_page_table && P_d > max_prefix_pages * ORACLE_PAGE) { bad = 1; continue; }
    /* K and V of prefix key j: a row of prefix_k / prefix_v, or a page slot */
    const uint16_t *pk_base = prefix_page_table ? k_cache : prefix_k;
    const uint16_t *pv_base = prefix_page_table ? v_cache : prefix_v;
#define PREFIX_ROW(j)                                                              \
  (prefix_page_table                                                               \
       ? (long)prefix_page_table[(long)d * max_prefix_pages + (j) / ORACLE_PAGE] * \
                 ORACLE_PAGE + (j) % ORACLE_PAGE                                   \
       : (long)prefix_cu[d] + (j))
    int bad_page = 0;
    if (prefix_page_table)
      for (int pp = 0; pp * ORACLE_PAGE < P_b; ++pp) {
        const int page = prefix_page_table[(long)d * max_prefix_pages + pp];
        if (page < 0 || page >= num_pages) bad_page = 1;
      }
    if (bad_page) { bad = 1; continue; }
    const int L_b = branch_len[b];
    if (L_b < 0 || L_b > max_pages * ORACLE_PAGE) { bad = 1; continue; }

    const int n_keys_max = P_b + L_b;
    /* scores of the visible keys, in visiting order */
    double *s = (double *)malloc(sizeof(double) * (size_t)(n_keys_max > 0 ? n_keys_max : 1));
    if (!s) { bad = 1; continue; }

    for (int i = 0; i < m; ++i) {
      const long row = (long)b * m + i;
      const uint16_t *qv = q + (row * H_q + h) * (long)D;
      double *o = out + (row * H_q + h) * (long)D;
      const int last_private = L_b - m + i; /* inclusive */
      int n = 0;

      /* visible prefix keys */
      for (int j = 0; j < P_b; ++j) {
        const uint16_t *kv = pk_base + (PREFIX_ROW(j) * H_kv + g) * D;
        double dot = 0.0;
        for (int c = 0; c < D; ++c) dot += bf16_to_double(qv[c]) * bf16_to_double(kv[c]);
        s[n++] = scale * dot;
      }
      /* visible private keys */
      for (int j = 0; j <= last_private; ++j) {
        const int page = page_table[(long)b * max_pages + j / ORACLE_PAGE];
        if (page < 0 || page >= num_pages) { bad = 1; continue; }
        const uint16_t *kv =
            k_cache + (((long)page * ORACLE_PAGE + j % ORACLE_PAGE) * H_kv + g) * D;
        double dot = 0.0;
        for (int c = 0; c < D; ++c) dot += bf16_to_double(qv[c]) * bf16_to_double(kv[c]);
        s[n++] = scale * dot;
      }

      if (n == 0) {
        for (int c = 0; c < D; ++c) o[c] = 0.0;
        lse[row * H_q + h] = -INFINITY;
        continue;
      }
      double M = -INFINITY;
      for (int t = 0; t < n; ++t) M = s[t] > M ? s[t] : M;
      double denom = 0.0;
      for (int t = 0; t < n; ++t) denom += exp(s[t] - M);
      for (int c = 0; c < D; ++c) o[c] = 0.0;

      /* second walk over the same visible keys, in the same order */
      int t = 0;
      for (int j = 0; j < P_b; ++j, ++t) {
        const uint16_t *vv = pv_base + (PREFIX_ROW(j) * H_kv + g) * D;
        const double w = exp(s[t] - M) / denom;
        for (int c = 0; c < D; ++c) o[c] += w * bf16_to_double(vv[c]);
      }
      for (int j = 0; j <= last_private; ++j) {
        const int page = page_table[(long)b * max_pages + j / ORACLE_PAGE];
        if (page < 0 || page >= num_pages) continue;
        const uint16_t *vv =
            v_cache + (((long)page * ORACLE_PAGE + j % ORACLE_PAGE) * H_kv + g) * D;
        const double w = exp(s[t] - M) / denom;
        for (int c = 0; c < D; ++c) o[c] += w * bf16_to_double(vv[c]);
        ++t;
      }
      lse[row * H_q + h] = M + log(denom);
    }
    free(s);
#undef PREFIX_ROW
  }
  return bad ? -1 : 0;
}

/*
 * Greedy P-MTP acceptance, item 2 above.
 * logits [B][m][V] bf16, drafts [B][m] -> out_tokens [B][m], accepted_len [B].
 */
void oracle_pmtp_accept(const uint16_t *logits, const int32_t *drafts, int B,
                        int m, int V, int32_t *out_tokens,
                        int32_t *accepted_len) {
  for (int b = 0; b < B; ++b) {
    for (int j = 0; j < m; ++j) {
      const uint16_t *row = logits + ((long)b * m + j) * (long)V;
      int best = 0;
      double best_val = -INFINITY;
      int seen = 0; /* a non-NaN value has been taken */
      for (int v = 0; v < V; ++v) {
        const double x = bf16_to_double(row[v]);
        if (isnan(x)) continue;
        if (!seen || x > best_val) {
          best = v;
          best_val = x;
          seen = 1;
        }
      }
      out_tokens[(long)b * m + j] = best;
    }
    int k = 0;
    while (k < m && drafts[(long)b * m + k] == out_tokens[(long)b * m + k]) ++k;
    accepted_len[b] = k;
  }
}
