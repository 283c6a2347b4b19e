/*
 * budgetdraft.h - C ABI of the speculative-step attention library (libbudgetdraft.so).
 *
 * One speculative step of BudgetDraft (arXiv 2606.00144, Algorithm 2) spends its
 * KV-cache attention in three places, each an entry point below, plus the merge they
 * share:
 *   bd_select_budget  builds the drafter's sparse view K_S^sp(B) under a KV budget B
 *                     (Sec. 3.4 TopKChunks; Algorithm 2, sparsify);
 *   bd_draft_attn     one of the gamma drafter decode passes over that view
 *                     (Algorithm 2, Draft);
 *   bd_verify_attn    the verifier's (gamma+1)-query pass over the full cache with a
 *                     causal mask inside the draft block (Algorithm 2, Verify);
 *   bd_combine        the log-sum-exp merge of attention computed over disjoint key
 *                     sets (split-K partials).
 * and its greedy acceptance in two more:
 *   bd_argmax         the arg max token of logits rows (Eq. accept);
 *   bd_accept         the longest agreeing prefix plus the verifier's bonus token
 *                     (Algorithm 2, accept);
 * and the cache update around it in two more:
 *   bd_write_block_rows  writes the block's new K/V rows into the caches;
 *   bd_advance        slides the observation window over the settled block rows and
 *                     appends their positions to the sparse view (Algorithm 2, Update).
 * Around them: bd_workspace_size / bd_workspace_status (scratch and device-side
 * errors), bd_draft_attn_static / bd_draft_static_status (bd_draft_attn without a
 * workspace, and its error word),
 * bd_check_wait_timeout (runs the device-side error path on purpose) and bd_strerror.
 *
 * Conventions shared by every call
 *   - All tensor arguments are DEVICE pointers owned by the caller (the row sources
 *     of bd_write_block_rows may also be pinned host memory); the library never
 *     allocates, frees or keeps a pointer after a call returns.
 *   - bf16 tensors are IEEE bfloat16 (raw 16-bit), fp32 are IEEE float, int32 are
 *     int32_t.  Every tensor is dense row-major in the order written.  bf16 tensors
 *     (caches, queries, outputs) and fp32 split-K partials must be 16-byte aligned;
 *     other fp32 and int32 tensors 4-byte aligned; logits passed to bd_argmax need
 *     only their element alignment.
 *   - KV caches are bf16 [batch, h_kv, t_cap, head_dim].  Rows hold post-RoPE keys
 *     and values: position p of (sequence b, KV head g) is row p.  Positions
 *     [0, t_ctx) are the context; rows t_ctx, t_ctx+1, ... hold the tokens of the
 *     current draft / verify block.
 *   - GQA: query head h reads KV head h / (h_q / h_kv).
 *   - Softmax scale is 1/sqrt(head_dim); every lse is a natural logarithm.
 *   - Calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy default
 *     stream).  A call returns BD_OK or a negative bd_status after validating every
 *     argument on the host BEFORE any launch; a failed launch returns BD_ERR_CUDA.
 *   - Workspace: `ws` is a caller-owned device buffer of at least
 *     bd_workspace_size(...) bytes for that call.  It must be zero-filled once
 *     before its first use; calls that finish leave its counter words zero again,
 *     so it can be reused without clearing.  Calls that share one workspace must
 *     be ordered (same stream, or synchronised).  Kernels record device-side
 *     errors (a bounded wait that ran out) in the workspace's status word, which
 *     bd_workspace_status() reads.
 *   - Supported: head_dim 64 or 128; h_q % h_kv == 0.
 */
#ifndef BUDGETDRAFT_H
#define BUDGETDRAFT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum bd_status {
  BD_OK = 0,
  BD_ERR_INVALID_ARG = -1,  /* a null pointer, a size out of range, inconsistent shape  */
  BD_ERR_UNSUPPORTED = -2,  /* valid but not implemented (head_dim, too many queries)    */
  BD_ERR_MISALIGNED = -3,   /* a tensor pointer lacks the alignment its call requires    */
  BD_ERR_WORKSPACE = -4,    /* ws is NULL or smaller than bd_workspace_size()            */
  BD_ERR_CUDA = -5,         /* a CUDA runtime call or a launch failed                    */
  BD_ERR_TIMEOUT = -6       /* device side: a bounded wait ran out (status word only)    */
} bd_status;

/* Problem shape of one layer's cache.  The caches are [batch, h_kv, t_cap, head_dim].
 * seq_lens (optional) gives every sequence its own context length T_b: a DEVICE int32
 * array [batch] with 1 <= T_b <= t_ctx, read by the kernels (so a step's lengths can be
 * advanced on the device by bd_advance); t_ctx is then the longest length and sizes the
 * launches.  Everything this header says of t_ctx holds per sequence with T_b in its
 * place.  NULL: every sequence has t_ctx.  A T_b outside [1, t_ctx] is recorded in the
 * workspace status word (BD_ERR_INVALID_ARG) and clamped into range.  With seq_lens,
 * batch * h_kv must not exceed 4096, and a call whose kernel keeps a table of
 * batch * h_kv + 1 ints in shared memory (the selection's score pass, the verify pass)
 * reports BD_ERR_UNSUPPORTED when that table does not fit beside its tiles (the verify
 * pass with 24 query rows per KV head holds about 2500). */
typedef struct bd_shape {
  int32_t batch;     /* sequences                                   */
  int32_t h_q;       /* query heads                                 */
  int32_t h_kv;      /* KV heads, divides h_q                        */
  int32_t head_dim;  /* d: 64 or 128                                 */
  int32_t t_ctx;     /* context length T (cached prefix positions)   */
  int32_t t_cap;     /* rows per (sequence, KV head) in the arrays   */
  const int32_t* seq_lens;  /* per-sequence lengths [batch] or NULL  */
} bd_shape;

/* Element types of bd_argmax logits. */
enum { BD_DTYPE_BF16 = 1, BD_DTYPE_F32 = 2 };

/* Operation codes for bd_workspace_size. */
enum { BD_OP_SELECT = 1, BD_OP_DRAFT = 2, BD_OP_VERIFY = 3 };

/*
 * Workspace bytes needed by one operation on `shape` (0 on invalid input).
 *   BD_OP_SELECT: budget = B, n_q = window W (window queries per head);
 *   BD_OP_DRAFT:  budget = B, n_q = the largest step_j + 1 that will be passed;
 *   BD_OP_VERIFY: budget ignored, n_q = queries per head in the block.
 * The size depends on the current device's SM count.  Sizes for different ops may
 * be satisfied by one buffer of the largest of them.
 */
size_t bd_workspace_size(const bd_shape* shape, int op, int budget, int n_q);

/* bd_select_budget flags. */
enum {
  /* q_window, window_lse and the shape's per-sequence lengths (if any) were written
   * before the kernel that immediately precedes this call on `stream` (not by it:
   * bd_advance, for one, rewrites all three in place): the call may read them while
   * that kernel finishes. */
  BD_SELECT_WINDOW_READY = 1
};

/*
 * KV-budget selection: the sparse drafter view K_S^sp(B) of every (sequence, KV
 * head).  Sec. 3.4 of the paper keeps the top floor(B/s) chunks of the prefix by
 * cumulative attention weight; this library reads "cumulative attention weight" of
 * position k as
 *     score[k] = sum over the group's query heads h and window rows w with k <= p_w
 *                of exp(q_{h,w} . k_k / sqrt(d) - lse_{h,w}),
 * the summed causal softmax probability that the last W context queries (window
 * row w sits at position p_w = t_ctx - W + w) put on key k.
 *   keep = [0, n_sink)  U  [t_ctx - n_recent, t_ctx)
 *          U  best of the middle [n_sink, t_ctx - n_recent):
 *               chunk == 1: the top (budget - n_sink - n_recent) positions by score;
 *               chunk == s > 1: the top floor((budget - n_sink - n_recent)/s) chunks,
 *                 chunk c = positions [c s, c s + s) within the middle, scored by the
 *                 sum of its members;
 *          ties go to the lower position (chunk).  If budget >= t_ctx, keep = [0, t_ctx).
 *
 *   k_cache     bf16 [batch, h_kv, t_cap, d]; rows [0, t_ctx) are read.
 *   q_window    bf16 [batch, h_q, window, d]: queries of positions t_ctx-W .. t_ctx-1.
 *   window_lse  fp32 [batch, h_q, window]: each window row's softmax normaliser over
 *               keys [0, p_w] (carried from the step that verified that token), or
 *               NULL to have it computed here (reads K a second time).
 *   flags       0 or BD_SELECT_WINDOW_READY.
 *   idx_out     int32 [batch, h_kv, budget]: kept positions ascending, then -1 padding.
 *   count_out   int32 [batch, h_kv]: number of kept positions.
 * Constraints: 1 <= window <= t_ctx, (h_q/h_kv)*window <= 256 (<= 128 with window_lse
 * NULL), n_sink, n_recent >= 0,
 * n_sink + n_recent <= budget when budget < t_ctx, chunk >= 1, t_cap >= t_ctx.
 */
int bd_select_budget(const bd_shape* shape, const void* k_cache, const void* q_window,
                     const float* window_lse, int window, int budget, int n_sink, int n_recent,
                     int chunk, unsigned flags, int32_t* idx_out, int32_t* count_out, void* ws,
                     size_t ws_bytes, void* stream);

/* bd_draft_attn flags. */
enum {
  /* idx, count and the context rows [0, t_ctx) of the caches were written before the
   * kernel that immediately precedes this call on `stream` (true for every pass after the
   * first of a speculative step): the call may start gathering them while that kernel
   * finishes.  The queries and the drafted rows are always read after it. */
  BD_DRAFT_VIEW_READY = 1
};

/*
 * Drafter decode pass j (0-based) over the sparse view (Algorithm 2, Draft):
 * each query head h of sequence b attends to rows idx[b, g, 0:count[b, g]] and to
 * the drafted rows t_ctx .. t_ctx + step_j of its KV head g (the drafter's own
 * tokens are appended to its sparse cache, Algorithm 2, Update).
 *   q        bf16 [batch, h_q, d]
 *   idx      int32 [batch, h_kv, budget] positions in [0, t_ctx) (as written by
 *            bd_select_budget; entries past count are ignored); count int32 [batch, h_kv]
 *            with 0 <= count <= budget.
 *   flags    0 or BD_DRAFT_VIEW_READY.
 *   o_out    bf16 [batch, h_q, d];  lse_out fp32 [batch, h_q] (may be NULL).
 * Constraints: step_j >= 0, t_ctx + step_j < t_cap, h_q / h_kv <= 16.  The budget + step_j + 1
 * entries are split over at most 8 CTAs, each holding the row table of its slice in shared
 * memory beside its tiles: at head_dim 128 views of up to about 165K (GQA group 16) to
 * 290K (group 1) entries, fewer when batch * h_kv fills the GPU; a larger view returns
 * BD_ERR_UNSUPPORTED.
 */
int bd_draft_attn(const bd_shape* shape, const void* q, const void* k_cache, const void* v_cache,
                  const int32_t* idx, const int32_t* count, int budget, int step_j, unsigned flags,
                  void* o_out, float* lse_out, void* ws, size_t ws_bytes, void* stream);

/*
 * bd_draft_attn without a workspace.  The paper has no counterpart: this entry point
 * exists for callers that cannot allocate device memory when they call the library,
 * for example a plugin that is handed only a stream and tensor pointers by its host
 * framework, or a serving loop whose device memory is fixed after start-up and which
 * must not call cudaMalloc between steps.  Such callers cannot supply the workspace that
 * bd_draft_attn needs.
 *
 * Arguments and results are those of bd_draft_attn with flags = 0, minus ws and ws_bytes.  The call
 * allocates nothing: its scratch (status word and per-(sequence, KV head) counters; the
 * drafter's split-K partials are merged inside each thread-block cluster) is a 4 MiB
 * array inside the library's device image, which every GPU
 * that loads the library keeps until the process exits.  A shape whose scratch would not
 * fit returns BD_ERR_WORKSPACE before any launch.
 *   - The first call on a device looks up that array's device address with the device
 *     current (cudaGetSymbolAddress); make that first call before any stream capture.
 *     The address is kept for the life of the process: after cudaDeviceReset on a device
 *     this entry point has been called on, it must not be called on that device again.
 *   - Every call clears the array's counters on `stream` before its kernel.  Device-side
 *     errors (an index outside the context, which is skipped as in bd_draft_attn) set the
 *     array's status word, which keeps them until bd_draft_static_status reads it.
 *   - All calls share the one array: calls whose work can overlap on the GPU (different
 *     streams, or threads without ordering between them) race and corrupt each other's
 *     results.  Issue them on one stream.
 */
int bd_draft_attn_static(const bd_shape* shape, const void* q, const void* k_cache,
                         const void* v_cache, const int32_t* idx, const int32_t* count, int budget,
                         int step_j, void* o_out, float* lse_out, void* stream);

/*
 * Status word of bd_draft_attn_static's array on the current device (no counterpart in
 * the paper): waits for `stream`, returns the first device-side error the calls on it
 * recorded since the last read (BD_OK if none) and clears it.  Call it on the stream
 * the static calls were issued on.
 */
int bd_draft_static_status(void* stream);

/*
 * Verifier block attention (Algorithm 2, Verify): query i (0 <= i < n_q) of head h
 * sits at position t_ctx + i and attends to keys [0, t_ctx + i] of its KV head.
 *   q        bf16 [batch, h_q, n_q, d]
 *   o_out    bf16 [batch, h_q, n_q, d], or NULL to compute lse only (V not read);
 *   lse_out  fp32 [batch, h_q, n_q] (may be NULL when o_out is not).
 * Constraints: 1 <= n_q, t_ctx + n_q <= t_cap, (h_q/h_kv)*n_q <= 768 (<= 128 when
 * o_out is NULL).  A KV head's query rows beyond 96 are processed in up to eight chunks
 * of equal size that stream the same keys side by side.
 */
int bd_verify_attn(const bd_shape* shape, const void* q, int n_q, const void* k_cache,
                   const void* v_cache, void* o_out, float* lse_out, void* ws, size_t ws_bytes,
                   void* stream);

/*
 * Log-sum-exp merge of attention over disjoint key sets: with L = log sum_s exp(lse_s),
 *   o = sum_s exp(lse_s - L) o_s,   lse = L.
 * A part with lse = -inf is empty and contributes nothing; rows whose parts are all
 * empty give o = 0 and lse = -inf.
 *   o_part   fp32 [n_split, rows, d], each row normalised over its own key set;
 *   lse_part fp32 [n_split, rows];
 *   o_out    bf16 [rows, d];  lse_out fp32 [rows] (may be NULL).
 * Constraints: 1 <= n_split <= 12288 (the merge weights of a row live in 48 KB of
 * shared memory; more parts return BD_ERR_UNSUPPORTED), rows >= 0 (0 is a no-op),
 * head_dim 64 or 128.
 */
int bd_combine(const float* o_part, const float* lse_part, int n_split, int rows, int head_dim,
               void* o_out, float* lse_out, void* stream);

/*
 * Greedy token choice (Eq. accept: a drafter token is accepted when it equals the
 * verifier's arg max at the same position): ids_out[r] = arg max over v of
 * logits[r, v].  Values are compared exactly in the stored type; ties go to the lowest
 * v, NaN is never chosen, -0 equals +0, and a row without a comparable value (all NaN)
 * gives 0.
 *   logits   bf16 or fp32 [rows, vocab] as `dtype` says (BD_DTYPE_*);
 *   ids_out  int32 [rows].
 * Constraints: 0 <= rows <= 65535 (0 is a no-op), 1 <= vocab <= 2^30.  No workspace.
 */
int bd_argmax(const void* logits, int dtype, int rows, int vocab, int32_t* ids_out, void* stream);

/*
 * Greedy acceptance of one speculative block (Algorithm 2, accept and bonus token):
 * k = the largest count with draft_tokens[i, b] == verify_tokens[b, i] for every
 * i < k (0 <= k <= gamma); the step emits those k drafter tokens followed by the
 * verifier's token verify_tokens[b, k].
 *   draft_tokens   int32 [gamma, batch]: the drafter's tokens x_hat, pass-major (row j
 *                  holds pass j's token of every sequence, as bd_argmax writes them one
 *                  pass at a time); may be NULL when gamma == 0;
 *   verify_tokens  int32 [batch, gamma + 1]: the verifier's arg max at each block
 *                  position, the last one past the block;
 *   n_accept_out   int32 [batch]: k (may be NULL);
 *   emit_out       int32 [batch, gamma + 1]: the k + 1 emitted tokens, then -1 padding
 *                  (may be NULL, not both).
 * Constraints: batch >= 0 (0 is a no-op), gamma >= 0.  No workspace.
 */
int bd_accept(int batch, int gamma, const int32_t* draft_tokens, const int32_t* verify_tokens,
              int32_t* n_accept_out, int32_t* emit_out, void* stream);

/*
 * Cache update after acceptance (Algorithm 2, Update).  The verify block held positions
 * t_ctx .. t_ctx + n_q - 1 (the token the step started from, then the drafts); after
 * acceptance of k_b drafts, sequence b's rows t_ctx .. t_ctx + k_b are settled, a_b =
 * clamp(n_accept[b], 0, n_q - 1) + 1 rows.  The K/V rows of the block were written into
 * the caches before bd_verify_attn and stay where they are.
 *   - Per-sequence lengths (shape->seq_lens set): sequence b advances by its own a_b, and
 *     this call adds a_b to seq_lens[b] on the device (the array is updated in place).
 *   - One shared length (seq_lens NULL): the batch advances by a = min_b a_b (every
 *     sequence stays on tokens its verifier confirmed); the caller uses t_ctx + a as the
 *     next step's t_ctx.
 * This call updates the state that carry-mode selection and the drafter need:
 *   - q_window / window_lse slide by a: they hold positions t_ctx + a - W ..
 *     t_ctx + a - 1 afterwards, the new rows taken from q_verify / verify_lse (the
 *     verifier's softmax normaliser of a block row IS that row's causal window LSE);
 *   - idx / count (optional): positions t_ctx .. t_ctx + a - 1 are appended to every
 *     unit's view (Algorithm 2 appends accepted tokens to the sparse cache); a unit
 *     whose view has no room (count + a > idx_capacity) is left unchanged.
 * (with per-sequence lengths, read T_b for t_ctx and a_b for a in both items.)
 *   n_accept      int32 [batch] accepted drafts per sequence (bd_accept's n_accept_out);
 *   q_verify      bf16 [batch, h_q, n_q, d]; verify_lse fp32 [batch, h_q, n_q] (NULL
 *                 together with window_lse);
 *   q_window      bf16 [batch, h_q, window, d], window_lse fp32 [batch, h_q, window]:
 *                 read and rewritten in place;
 *   idx           int32 [batch, h_kv, idx_capacity], count int32 [batch, h_kv] (both
 *                 NULL to skip the view);
 *   advance_out   int32 [batch]: each sequence's advance (may be NULL).
 * Constraints: 1 <= window <= t_ctx, 1 <= n_q, t_ctx + n_q <= t_cap.  No workspace.
 */
int bd_advance(const bd_shape* shape, int window, int n_q, const int32_t* n_accept, const void* q_verify,
               const float* verify_lse, void* q_window, float* window_lse, int32_t* idx, int32_t* count,
               int idx_capacity, int32_t* advance_out, void* stream);

/*
 * Writes the K/V rows of the current block into the caches: rows t_ctx .. t_ctx + n_rows - 1
 * of every (sequence, KV head) (Algorithm 2, Update: new tokens' keys and values join the
 * cache).  Two strided copies on `stream` (cudaMemcpy2DAsync with cudaMemcpyDefault), or with
 * per-sequence lengths one kernel that writes rows T_b .. T_b + n_rows - 1; the sources may
 * be device memory or pinned host memory either way.
 *   k_rows, v_rows  bf16 [batch, h_kv, n_rows, d], dense;
 *   k_cache, v_cache bf16 [batch, h_kv, t_cap, d].
 * Constraints: 1 <= n_rows, t_ctx + n_rows <= t_cap.  No workspace.
 */
int bd_write_block_rows(const bd_shape* shape, int n_rows, const void* k_rows, const void* v_rows, void* k_cache,
                        void* v_cache, void* stream);

/*
 * Diagnostic of the device-side error path (the paper has no counterpart): launches one
 * small kernel that waits on a shared-memory barrier nothing completes, gives up after
 * limit_us microseconds (1 .. 2000000) like every bounded wait in the library, records
 * BD_ERR_TIMEOUT in the workspace's status word and returns; a second warp waiting on the
 * same barrier stops through the shared abort flag, as the roles of a pipelined kernel do.
 * No fault, trap or hang: the context stays usable, and bd_workspace_status() then reads
 * BD_ERR_TIMEOUT.  ws needs only the 256-byte status header.
 */
int bd_check_wait_timeout(void* ws, size_t ws_bytes, int limit_us, void* stream);

/*
 * Reads (and clears) the device status word of a workspace: BD_OK, or the first
 * device-side error recorded by a kernel since the last read.  Synchronises
 * `stream`.  Returns BD_ERR_INVALID_ARG for a NULL ws, BD_ERR_CUDA if the copy fails.
 */
int bd_workspace_status(void* ws, void* stream);

/* Static description of a status code. */
const char* bd_strerror(int status);

#ifdef __cplusplus
}
#endif

#endif /* BUDGETDRAFT_H */
