/*
 * hpd.h -- C ABI of libhpd, the GB300 (sm_103a) branch-decode step of
 * Hierarchical Parallel Decoding (HPD-Parsing).
 *
 * One call of hpd_branch_attn is the attention of one decoder layer for one
 * decode step of many concurrent content branches.  A content branch is
 * forked from the layout branch of its page and attends to
 *   - the page's shared prefix (the vision tokens plus the layout branch's
 *     tokens up to the fork position), whose KV is reused, never recomputed,
 *     and
 *   - its own private KV history only, never that of another branch
 * (Sec. 3.3, "Dynamic Branch Forking and Efficient Context Isolation").
 * Each branch carries m P-MTP query tokens that are causal among themselves
 * (Sec. 3.4, "Integration with P-MTP").  hpd_pmtp_accept is the greedy
 * verification of the P-MTP drafts that follows the forward pass (Sec. 3.4;
 * the verification step of Algorithm 1).
 *
 * Conventions for every entry point
 *   - Every pointer named in an argument list or struct is DEVICE memory of
 *     the current device, owned by the caller; the library keeps no pointer
 *     after the call returns.  Nothing here allocates, frees or synchronises
 *     (except hpd_read_errors, which says so).
 *   - Work is enqueued on `stream` (a cudaStream_t; NULL = legacy default
 *     stream) and runs asynchronously.
 *   - Host-side scalars are validated before anything is launched; a bad
 *     value returns HPD_ERR_INVALID_ARG / HPD_ERR_UNSUPPORTED and launches
 *     nothing.  Device-side integer arrays (offsets, lengths, page ids) are
 *     not read by the host: the kernels clamp every such value into range
 *     and record what they clamped in the workspace's error word (see
 *     hpd_read_errors), so no device content can make a kernel access memory
 *     outside the buffers described here.
 *   - A failed launch returns HPD_ERR_CUDA; hpd_last_cuda_error() gives the
 *     CUDA error code of the most recent failure on the calling thread.
 *   - bf16 means IEEE bfloat16, stored as 2-byte little-endian words.
 */
#ifndef HPD_H_
#define HPD_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st *hpd_stream_t; /* identical to cudaStream_t */

typedef enum {
  HPD_OK = 0,
  HPD_ERR_INVALID_ARG = 1, /* a host scalar or pointer is out of contract */
  HPD_ERR_UNSUPPORTED = 2, /* a legal shape the library has no kernel for */
  HPD_ERR_WORKSPACE = 3,   /* workspace missing, misaligned or too small */
  HPD_ERR_CUDA = 4,        /* a CUDA runtime call or launch failed */
  HPD_ERR_TIMEOUT = 5      /* a bounded device-side wait gave up */
} hpd_status;

/* Bits of the workspace error word (sticky until hpd_workspace_init). */
#define HPD_DEVERR_PREFIX_CU 0x1u   /* prefix_cu not monotone / beyond prefix_tokens */
#define HPD_DEVERR_BRANCH_CU 0x2u   /* branch_cu not monotone / beyond B */
#define HPD_DEVERR_BRANCH_LEN 0x4u  /* branch_len < 0 or > 16 * max_pages_per_branch */
#define HPD_DEVERR_PAGE_ID 0x8u     /* a page id outside [0, num_pages) */
#define HPD_DEVERR_FORK_LEN 0x10u   /* branch_prefix_len < 0 or > P_d */
#define HPD_DEVERR_TIMEOUT 0x40u    /* a bounded device-side wait expired */
#define HPD_DEVERR_POOL 0x80u       /* KV append / rollback: free-page stack short or inconsistent */
#define HPD_DEVERR_FORK_CAP 0x100u  /* fork: more branches than the output capacity */

/* Tokens per KV page of the paged private cache. */
#define HPD_PAGE_TOKENS 16

/*
 * Arguments of one branch-attention step.
 *
 * Notation: n_docs pages (documents); page d owns branches
 * [branch_cu[d], branch_cu[d+1]) and the prefix tokens
 * [prefix_cu[d], prefix_cu[d+1]) of prefix_k / prefix_v, so P_d =
 * prefix_cu[d+1] - prefix_cu[d].  Branch b has L_b = branch_len[b] private
 * KV entries, which INCLUDE the K/V of this step's m query tokens (they are
 * written to the cache before the call).  G = H_q / H_kv query heads share
 * one KV head; query head h reads KV head h / G.
 *
 * Query i (0 <= i < m) of branch b sees
 *   prefix keys  j <  P_b   (P_b = branch_prefix_len[b] if given, else P_d)
 *   private keys j <= L_b - m + i
 * Private key j is slot j % 16 of physical page page_table[b][j / 16].
 * The prefix is contiguous (prefix_k / prefix_v rows), or, when
 * prefix_page_table is set, paged in the same pool: prefix token j of page d
 * is slot j % 16 of physical page prefix_page_table[d][j / 16], shared by all
 * of the page's branches without a copy (Algorithm 1: a forked branch shares
 * its parent's KV pages; Sec. 3.3).
 * S_j = scale * <q, k_j>; out = softmax(S) V over the visible keys;
 * lse = ln sum_j exp(S_j).  No visible key: out = 0, lse = -inf.
 *
 * Alignment: q, prefix_k, prefix_v, k_cache, v_cache and out 16-byte aligned
 * (a 32-byte aligned out is written with 32-byte stores), lse and the int32
 * arrays 4-byte aligned, workspace 256-byte aligned; otherwise
 * HPD_ERR_INVALID_ARG (HPD_ERR_WORKSPACE for the workspace).
 */
typedef struct {
  const void *q;        /* bf16 [B*m][H_q][D]; row b*m + i                        */
  const void *prefix_k; /* bf16 [prefix_tokens][H_kv][D]                          */
  const void *prefix_v; /* bf16 [prefix_tokens][H_kv][D]                          */
  const int32_t *prefix_cu;         /* [n_docs+1], non-decreasing, <= prefix_tokens */
  const int32_t *branch_cu;         /* [n_docs+1], non-decreasing, branch_cu[n_docs] == B */
  const int32_t *branch_prefix_len; /* [B] fork-position prefix length, or NULL     */
  const void *k_cache;  /* bf16 [num_pages][16][H_kv][D]                           */
  const void *v_cache;  /* bf16 [num_pages][16][H_kv][D]                           */
  const int32_t *page_table;        /* [B][max_pages_per_branch]                    */
  const int32_t *branch_len;        /* [B], 0 <= L_b <= 16 * max_pages_per_branch   */
  int n_docs;               /* >= 1                                               */
  int B;                    /* >= 1 branches                                      */
  int m;                    /* 1..16 P-MTP query tokens per branch                */
  int H_q, H_kv;            /* H_q % H_kv == 0, G = H_q / H_kv <= 16               */
  int D;                    /* head dim: 64 or 128                                */
  int num_pages;            /* >= 1 pages in k_cache / v_cache                    */
  int max_pages_per_branch; /* >= 1 columns of page_table                         */
  int prefix_tokens;        /* rows of prefix_k / prefix_v (>= 0)                 */
  int max_prefix_len;       /* host upper bound on every P_d; 0 = prefix_tokens   */
  float scale;              /* softmax scale; 0 = 1/sqrt(D)                       */
  void *out;                /* bf16 [B*m][H_q][D]                                 */
  float *lse;               /* fp32 [B*m][H_q], natural log; may be NULL          */
  void *workspace;          /* 256-byte aligned, initialised once by
                               hpd_workspace_init; one call at a time per workspace */
  size_t workspace_bytes;
  /* Paged prefix (NULL: contiguous).  When set, prefix_k / prefix_v are not
   * read (may be NULL), prefix_cu still gives every P_d (only its differences
   * matter, bounded by prefix_tokens) and P_d <= 16 * max_prefix_pages, else
   * HPD_DEVERR_PREFIX_CU and the prefix is cut there.  A table entry outside
   * [0, num_pages) is flagged HPD_DEVERR_PAGE_ID and read as page 0; entries
   * past a page's last prefix page are not read. */
  const int32_t *prefix_page_table; /* [n_docs][max_prefix_pages]                 */
  int max_prefix_pages;             /* >= 1 columns when prefix_page_table is set */
} hpd_branch_attn_args;

/* Bytes of workspace hpd_branch_attn needs for these host scalars (the
 * device pointers in args are not read).  Returns 0 if the scalars are
 * invalid. */
size_t hpd_branch_attn_workspace_size(const hpd_branch_attn_args *args);

/* Zero the workspace (error word and arrival tickets) on `stream`.  Call
 * once after allocating it; every hpd_branch_attn call leaves the tickets
 * at zero again, so the workspace stays reusable. */
hpd_status hpd_workspace_init(void *workspace, size_t workspace_bytes, hpd_stream_t stream);

/* The branch-decode attention step (see the struct above).  Enqueues its
 * kernels on `stream`; out / lse are complete when the stream reaches that
 * point.  Concurrent calls must use distinct workspaces. */
hpd_status hpd_branch_attn(const hpd_branch_attn_args *args, hpd_stream_t stream);

/* Number of kernels one hpd_branch_attn call launches for these scalars
 * (0 if they are invalid).  When H_q / H_kv divides 128 the step runs on
 * tcgen05 tensor cores: one persistent kernel for the shared prefix and the
 * private suffixes, preceded by a one-CTA pass that orders its work units
 * longest first when there are at least two units per SM, and followed by a
 * merge kernel when the keys are split across CTAs.
 * Otherwise: a warp-MMA shared-prefix kernel, then a warp-MMA private-suffix
 * kernel that also merges and writes out / lse. */
int hpd_branch_attn_launches(const hpd_branch_attn_args *args);

/* Name of the k-th of those kernels (static string), or NULL. */
const char *hpd_branch_attn_kernel_name(const hpd_branch_attn_args *args, int k);

/* hpd_branch_attn with timing markers.  stage_events holds
 * hpd_branch_attn_launches(args) + 1 cudaEvent_t handles created by the
 * caller (with timing enabled); event 0 is recorded on `stream` before the
 * first kernel and event k after the k-th.  While `stream` is capturing they
 * are recorded as external event nodes (so a replayed graph times each
 * kernel), otherwise as plain records.  NULL behaves as hpd_branch_attn. */
hpd_status hpd_branch_attn_marked(const hpd_branch_attn_args *args, hpd_stream_t stream,
                                  void *const *stage_events);

/*
 * Greedy P-MTP verification (Sec. 3.4; Algorithm 1, verification step).
 *   logits       bf16 [B][m][V]   target-model logits at the m draft positions
 *   drafts       int32 [B][m]     drafted tokens; drafts[b][j] is checked
 *                                 against the argmax of logits row j
 *   out_tokens   int32 [B][m]     t*_{b,j} = argmax_v logits[b][j][v], the
 *                                 lowest index among equal maxima; NaN never
 *                                 wins (an all-NaN row gives 0)
 *   accepted_len int32 [B]        n_acc_b = largest k <= m such that
 *                                 drafts[b][i] == t*_{b,i} for all i < k
 * The caller emits t*_{b,0 .. min(n_acc_b, m-1)}: the accepted drafts plus
 * the target's own token at the first mismatch.
 * Requires B >= 1, 1 <= m <= 64, V >= 1.
 */
hpd_status hpd_pmtp_accept(const void *logits, const int32_t *drafts, int B, int m, int V,
                           int32_t *out_tokens, int32_t *accepted_len, hpd_stream_t stream);

/*
 * One branch-decode step (Algorithm 1: the model step, then verification):
 * hpd_branch_attn(args) and hpd_pmtp_accept over logits [B][m][V] and drafts
 * [B][m] (B = args->B, m = args->m), with exactly the results of the two
 * calls made in that order on `stream`, and the same argument checks and
 * errors (nothing is enqueued when either call's arguments are refused).
 *
 * The acceptance reads only logits and drafts, none of the attention's
 * results, so the two need not run one after the other.  When the attention
 * kernel leaves SMs idle for part of its run (fewer than two work units per
 * SM: its persistent grid is smaller than the SM count, as on a one-page
 * step, or its last round of whole units leaves SMs idle) the acceptance
 * runs on those SMs while the attention runs: it is launched on a second
 * stream owned by the library,
 * forked from `stream` and joined back to it with events, so the step stays
 * ordered on `stream` (work enqueued on `stream` afterwards waits for both)
 * and can be captured in a CUDA graph.  Otherwise the acceptance follows the
 * attention on `stream`.  The second stream and its two events are created
 * on the first call made outside stream capture on each device (a call
 * inside capture before then runs the two in order).  Calls from several
 * host threads take a lock while they enqueue.  The second stream is shared
 * by every call on the device, so the acceptances of steps issued on
 * different streams run one after another.
 */
hpd_status hpd_decode_step(const hpd_branch_attn_args *args, const void *logits,
                           const int32_t *drafts, int V, int32_t *out_tokens,
                           int32_t *accepted_len, hpd_stream_t stream);

/* 1 when hpd_decode_step would run the acceptance concurrently with the
 * attention for these host scalars (device pointers are not read), 0 when
 * in order, -1 for invalid scalars or an unavailable device. */
int hpd_decode_step_concurrent(const hpd_branch_attn_args *args);

/*
 * hpd_branch_attn for callers that cannot allocate device memory.  The
 * paper has no counterpart to this entry point.
 *
 * Some callers of this library cannot obtain a workspace: a plugin whose
 * host engine owns all device memory and passes it only its inputs and
 * outputs, or code on a path where cudaMalloc (which can synchronise the
 * whole device) is not allowed.  This variant computes exactly what
 * hpd_branch_attn computes, but keeps its scratch in a file-scope device
 * array of HPD_NOALLOC_WORKSPACE_BYTES inside libhpd, which every GPU that
 * loads the library holds until the process exits.  args->workspace and
 * args->workspace_bytes are ignored (they may be NULL / 0); every other
 * field means what it means for hpd_branch_attn.
 *   - Nothing is allocated: no cudaMalloc, cudaFree or allocating library
 *     routine is called.
 *   - Every argument is checked as hpd_branch_attn checks it before
 *     anything is enqueued; a refused call touches neither the array nor
 *     the stream.  A shape whose hpd_branch_attn_workspace_size exceeds
 *     HPD_NOALLOC_WORKSPACE_BYTES is refused with HPD_ERR_WORKSPACE.
 *   - The first call on a device looks up the array's device address
 *     (cudaGetSymbolAddress, with that device current); make that first call
 *     before any stream capture on the device.
 *   - All calls share the one array, which keeps the previous call's
 *     contents; each call clears its error word on `stream` first.  Calls
 *     whose work overlaps on the GPU (other streams, other threads) race on
 *     the array and give undefined results: serialise them.
 *   - The clamp flags of the device-side checks are kept in the shared array
 *     and are not reported (hpd_read_errors needs a caller workspace).
 */
#define HPD_NOALLOC_WORKSPACE_BYTES (32u << 20)
hpd_status hpd_branch_attn_noalloc(const hpd_branch_attn_args *args, hpd_stream_t stream);

/* Copy the workspace error word (HPD_DEVERR_* bits) to *flags.  This is the
 * one call that synchronises: it waits for `stream`. */
hpd_status hpd_read_errors(const void *workspace, uint32_t *flags, hpd_stream_t stream);

/* ------------------------------------------------------------------------
 * Paged private KV around a decode step (Algorithm 1: the step's tokens are
 * written to the cache before attention -- WriteKV -- and after verification
 * the branch keeps what was accepted; the printed length update is garbled,
 * read here as "keep n_acc + 1 of the step's m rows, roll back the rest").
 *
 * Free pages live on a device stack: free_pages[0 .. *free_top) hold page ids
 * not used by any branch.  Logical page i of branch b is allocated exactly
 * when i < ceil(branch_len[b] / 16).  Allocation is deterministic (branch
 * order), all or nothing: on a short stack or a branch that would outgrow
 * max_pages * 16 rows, nothing changes and the workspace error word gets
 * HPD_DEVERR_POOL / HPD_DEVERR_BRANCH_LEN.  Device pointers; the caller owns
 * everything; calls are asynchronous on `stream`.
 * ------------------------------------------------------------------------ */
typedef struct {
  const void *k_new;    /* bf16 [B][m][H_kv][D]: the step's new keys (append) */
  const void *v_new;    /* bf16 [B][m][H_kv][D]: the step's new values (append) */
  void *k_cache;        /* bf16 [num_pages][16][H_kv][D], 16-byte aligned */
  void *v_cache;        /* bf16 [num_pages][16][H_kv][D], 16-byte aligned */
  int32_t *page_table;  /* [B][max_pages]; freed entries become -1 */
  int32_t *branch_len;  /* [B], updated in place */
  int32_t *free_pages;  /* [num_pages] stack of free page ids */
  int32_t *free_top;    /* [1] number of ids on the stack */
  void *workspace;      /* 256-byte aligned, >= 256 bytes; word 0: HPD_DEVERR_* bits
                           (cleared by the caller, e.g. hpd_workspace_init), word 1:
                           1 when the last append allocated */
  int B, m, H_kv, D;    /* m in 1..64, D in {64, 128} */
  int num_pages, max_pages;
} hpd_kv_args;

/* Append: branch b's m rows of k_new / v_new go to private positions
 * [L_b, L_b + m) (pages opened by them popped from the stack), L_b += m. */
hpd_status hpd_kv_append(const hpd_kv_args *args, hpd_stream_t stream);

/* Rollback after hpd_pmtp_accept (same stream): of the step's m rows at
 * [L_b - m, L_b), keep the first min(accepted_len[b] + 1, m) (none when
 * accepted_len[b] < 0); L_b shrinks accordingly and the pages past the new
 * length go back onto the stack in branch order.  accepted_len: int32 [B],
 * device.  k_new / v_new are not used. */
hpd_status hpd_kv_rollback(const hpd_kv_args *args, const int32_t *accepted_len,
                           hpd_stream_t stream);

/* ------------------------------------------------------------------------
 * Fork detection and child branches after verification (Algorithm 1: scan
 * the accepted tokens for the fork token, spawn a child sharing the parent's
 * context; Sec. 3.3).  A page's shared context is its prefix (vision tokens,
 * then its layout branch's tokens), so a child is a new branch of the same
 * page whose fork-position prefix length is just past the fork token, with
 * no private keys: nothing is copied.
 *
 * A layout branch b (is_layout[b] != 0, or every branch when is_layout is
 * NULL) emits out_tokens[b][0 .. e_b), e_b = min(accepted_len[b] + 1, m)
 * (accepted drafts, then the correction token); token i sits at prefix
 * position layout_pos[b] + i.  Each emitted fork token spawns a child with
 * prefix length layout_pos[b] + i + 1, private length 0 and an all -1 page
 * table row.  Outputs (device, capacity `cap` branches): the branch arrays of
 * the new set, each page's old branches first (in order), then its children
 * in (parent, index) order; new_parent[i] = the old index of an old branch,
 * or -1 - parent for a child; new_branch_prefix_len of an old branch is its
 * branch_prefix_len (-1 when that array is NULL: the whole page prefix).
 * *new_B = the new branch count, or -1 with HPD_DEVERR_FORK_CAP in the
 * workspace error word when it would exceed cap (the outputs are then not
 * written).  workspace: 256-byte aligned, >= 4 * (65 + n_docs) bytes, word 0
 * the error word (cleared by the caller).  One launch (B + n_docs up to
 * 11,998; two launches beyond), asynchronous on `stream`.
 * ------------------------------------------------------------------------ */
typedef struct {
  const int32_t *out_tokens;         /* [B][m] (hpd_pmtp_accept) */
  const int32_t *accepted_len;       /* [B] */
  const int32_t *is_layout;          /* [B] or NULL */
  const int32_t *layout_pos;         /* [B] prefix position of the step's token 0 */
  const int32_t *branch_cu;          /* [n_docs + 1], monotone, branch_cu[n_docs] = B */
  const int32_t *branch_prefix_len;  /* [B] or NULL */
  const int32_t *branch_len;         /* [B] */
  const int32_t *page_table;         /* [B][max_pages] */
  int32_t *new_branch_cu;            /* [n_docs + 1] */
  int32_t *new_branch_prefix_len;    /* [cap] */
  int32_t *new_branch_len;           /* [cap] */
  int32_t *new_page_table;           /* [cap][max_pages] */
  int32_t *new_parent;               /* [cap] */
  int32_t *new_B;                    /* [1] */
  void *workspace;
  size_t workspace_bytes;
  int32_t fork_token;
  int B, m, n_docs, max_pages, cap;
} hpd_fork_args;

hpd_status hpd_fork_children(const hpd_fork_args *args, hpd_stream_t stream);

/* Self-test of the bounded device waits (no counterpart in the paper): one
 * warp waits on an mbarrier phase that nothing completes and on a
 * shared-memory flag that nothing sets, each for about limit_us
 * microseconds (1 .. 10,000,000), then returns normally.  Each wait that gave
 * up sets a bit in the workspace error word: HPD_DEVERR_TIMEOUT for the
 * mbarrier and HPD_DEVERR_TIMEOUT << 8 for the flag.  workspace: device
 * pointer, 256-byte aligned, at least 256 bytes; the caller clears it first
 * (hpd_workspace_init) and reads it with hpd_read_errors.  Asynchronous on
 * `stream`; HPD_ERR_INVALID_ARG for a bad pointer or limit. */
hpd_status hpd_wait_selftest(void *workspace, uint32_t limit_us, hpd_stream_t stream);

/* Static description of a status code. */
const char *hpd_status_string(hpd_status status);

/* CUDA error code (cudaError_t value) of the last HPD_ERR_CUDA on this thread. */
int hpd_last_cuda_error(void);

/* Library version, major * 10000 + minor * 100 + patch. */
int hpd_version(void);

#ifdef __cplusplus
}
#endif
#endif /* HPD_H_ */
