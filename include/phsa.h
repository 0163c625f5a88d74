/*
 * phsa.h -- C ABI of the PHSA sparse-attention library for NVIDIA GB300 (sm_103a).
 *
 * PHSA (Punctuation-aware Hybrid Sparse Attention) replaces dense causal
 * attention by attention over a few selected key/value blocks. The library
 * implements its three stages as CUDA kernels:
 *   (a) phsa_build_block_repr  -- one representative key per KV block, mixing
 *       the block's mean key with the mean of its punctuation-token keys
 *       (Section 3.2, Eq. 3, 6, 7, 8; Algorithm 1 step 2);
 *   (b) phsa_select_blocks     -- query-to-block relevance and Top-K block
 *       selection with forced initial and local blocks (Eq. 8; Section 3.2
 *       "Block Selection"; Algorithm 1 step 3);
 *   (c) phsa_sparse_attn_fwd / phsa_sparse_attn_bwd -- causal attention over
 *       the selected blocks only (Eq. 10-11; Algorithm 1 step 4) and its
 *       gradient, which the paper's native sparse training uses.
 *
 * Conventions shared by every call
 *   - Tensors are dense, row-major, layout [B, H, L, D]; bf16 values are
 *     IEEE bfloat16 (uint16 storage). Query head h reads KV head h / G with
 *     G = Hq / Hkv (grouped-query attention).
 *   - Blocks have block_size = m tokens; block t covers tokens [t*m, (t+1)*m).
 *     T = floor(L/m) blocks have a representative key (Eq. 3); NQB = ceil(L/m)
 *     query blocks exist (the last may be partial).
 *   - Selection is shared by the G*m query rows of one (query block, KV head):
 *     block_idx[b][g][qb][0..cnt) lists block indices in ascending order,
 *     padded with -1 up to topk; block_cnt[b][g][qb] = cnt.
 *   - Every tensor pointer is a DEVICE pointer owned by the caller, 16-byte
 *     aligned. The library never frees or retains caller memory.
 *   - All work is enqueued on `stream` (a cudaStream_t passed as void*; NULL
 *     is the legacy default stream) and is asynchronous. The return value
 *     reports argument validation and launch errors only. Errors detected by
 *     a kernel (an out-of-range block index, a bounded wait that expired) are
 *     recorded in a device status word read by phsa_get_device_status.
 *   - Supported today: D = 128, G in {1, 2}, block_size 16, 32 or 64 (16 is
 *     the block size of the paper's experiment settings) in every call, with
 *     two exceptions: the backward (phsa_sparse_attn_bwd, its workspace query
 *     and the no-allocation entry point) takes 16 and 32 only for G = 2, and
 *     the host-buffer step (phsa_step_host) takes 64 only.
 *     Other shapes return PHSA_ERR_UNSUPPORTED, never a wrong answer.
 *   - Calls are thread-safe with respect to each other; concurrent calls on
 *     different streams that write the same output race, as any CUDA work.
 */
#ifndef PHSA_H
#define PHSA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    PHSA_OK = 0,
    PHSA_ERR_INVALID_ARG = -1,  /* null/misaligned pointer, bad size or parameter */
    PHSA_ERR_UNSUPPORTED = -2,  /* valid but unsupported shape (D, block_size, G) */
    PHSA_ERR_CUDA = -3,         /* a CUDA runtime call or launch failed */
    PHSA_ERR_TIMEOUT = -4,      /* device: a bounded wait inside a kernel expired */
    PHSA_ERR_DEVICE_INDEX = -5, /* device: a block index outside [0, qb] was skipped */
    PHSA_ERR_WORKSPACE = -6     /* workspace pointer null or smaller than required */
} phsa_status;

/* Problem shape. Layout [B, H, L, D]; block_size = m tokens per block. */
typedef struct {
    int B, L, Hq, Hkv, D, block_size;
} phsa_shape;

/* How the G*m query rows of a (query block, KV head) unit are combined into
 * one relevance A_t per candidate block t (the paper scores single tokens,
 * Eq. 8; the group rule is this library's reading):
 *   PHSA_AGG_SOFTMAX_SUM  A_t = sum over the rows of the row's softmax
 *                         probability of block t over the candidates (Eq. 8);
 *   PHSA_AGG_MAX_LOGIT    A_t = max over the rows of the raw score
 *                         q_r . Krepr_t * sm_scale (one pass, no softmax).
 * Both reduce to Algorithm 1's per-token ranking for a single row. */
#define PHSA_AGG_SOFTMAX_SUM 0
#define PHSA_AGG_MAX_LOGIT 1

/* Selection parameters (Algorithm 1 inputs k, n_init and w).
 *   topk        total blocks per (query block, KV head), forced blocks included
 *               (the paper's 32k setting of 128 initial + 512 local tokens plus
 *               16 chosen 16-token blocks is 896 tokens = 14 blocks of 64);
 *   n_init      forced initial blocks {0 .. n_init-1};
 *   n_local     forced local blocks {qb-n_local+1 .. qb}, n_local >= 1 (the
 *               query's own block is always attended);
 *   sm_scale    score scale, normally 1/sqrt(D) (Eq. 2, 8, 11);
 *   aggregation PHSA_AGG_SOFTMAX_SUM (0, the default of a zeroed struct) or
 *               PHSA_AGG_MAX_LOGIT; other values are PHSA_ERR_INVALID_ARG.
 * Requires topk >= n_init + n_local, so every query block's forced set fits. */
typedef struct {
    int topk, n_init, n_local;
    float sm_scale;
    int aggregation;
} phsa_select_params;

/*
 * Punctuation indicator, Section 3.2 Eq. 4-5: mask[i] = 1 if ids[i] is one of
 * the n_punct ids of the punctuation set P, else 0 (the set is given as ids,
 * in any order, duplicates allowed; building it from a vocabulary is the
 * caller's job).
 *   ids        int32 [n]        in (device)
 *   punct_ids  int32 [n_punct]  in (device), 0 <= n_punct <= 4096
 *   mask       uint8 [n]        out (device)
 * PHSA_ERR_UNSUPPORTED for n_punct > 4096; n = 0 does nothing.
 */
int phsa_punct_mask(const int32_t* ids, int64_t n, const int32_t* punct_ids, int n_punct,
                    uint8_t* mask, void* stream);

/*
 * Stage (a): representative keys, Section 3.2 Eq. 6-8 / Algorithm 1 step 2.
 * For every (b, g, t < T): M_0 = mean of the block's m keys (Eq. 6);
 * c = number of punctuation tokens in the block; M_p = mean of their keys if
 * c > 0 (Eq. 7), else M_0; Krepr = lambda*M_0 + (1-lambda)*M_p (Eq. 8).
 * Sums in fp32, one round-to-nearest-even to bf16 at the end.
 *   K          bf16 [B, Hkv, L, D]   in
 *   punct_mask uint8 [B, L]          in, nonzero = token is punctuation (I(x in P))
 *   lambda     gate in [0, 1]
 *   Krepr      bf16 [B, Hkv, T, D]   out (nothing is written when T = 0)
 */
int phsa_build_block_repr(const void* K, const uint8_t* punct_mask, phsa_shape s, float lambda,
                          void* Krepr, void* stream);

/*
 * Stage (b): relevance scoring and block selection, Eq. 8 / Algorithm 1 step 3,
 * made once per (query block qb, KV head g) for all G*m rows r of that block:
 *   forced   F = {0..n_init-1} U {qb-n_local+1..qb}, clipped to [0, qb];
 *   candidates C = {t <= qb-1, t < T, t not in F} (strictly earlier full blocks);
 *   S[r][t] = sm_scale * q_r . Krepr[t];  p[r][t] = softmax over t in C of S[r][.];
 *   A[t]    = sum over rows r of p[r][t];
 *   choose min(topk-|F|, |C|) candidates by A descending, ties to the lower t;
 *   output F U chosen in ascending order, -1 padded to topk.
 * Scores stay on chip (they are never written to memory).
 *   Q         bf16 [B, Hq, L, D]        in
 *   Krepr     bf16 [B, Hkv, T, D]       in (from phsa_build_block_repr)
 *   block_idx int32 [B, Hkv, NQB, topk] out
 *   block_cnt int32 [B, Hkv, NQB]       out
 */
int phsa_select_blocks(const void* Q, const void* Krepr, phsa_shape s, phsa_select_params p,
                       int32_t* block_idx, int32_t* block_cnt, void* stream);

/*
 * Stage (c) forward: Eq. 10-11 / Algorithm 1 step 4. Row i of query head h
 * attends the keys j of the listed blocks of (qb = i/m, g = h/G) with j <= i,
 * o_i = sum_j softmax_j(sm_scale * q_i . k_j) v_j; lse_i = natural-log
 * log-sum-exp of those scores (kept for the backward pass).
 * block_idx entries must satisfy -1 or 0 <= t <= qb; entries beyond block_cnt
 * are ignored. An entry outside that range is skipped and recorded as
 * PHSA_ERR_DEVICE_INDEX in the device status word.
 *   Q            bf16 [B, Hq, L, D]   in
 *   K, V         bf16 [B, Hkv, L, D]  in
 *   block_idx    int32 [B, Hkv, NQB, topk], block_cnt int32 [B, Hkv, NQB]  in
 *   O            bf16 [B, Hq, L, D]   out
 *   lse          fp32 [B, Hq, L]      out
 */
int phsa_sparse_attn_fwd(const void* Q, const void* K, const void* V, const int32_t* block_idx,
                         const int32_t* block_cnt, phsa_shape s, int topk, float sm_scale,
                         void* O, float* lse, void* stream);

/* Bytes of device workspace phsa_sparse_attn_bwd needs for this shape/topk. */
size_t phsa_sparse_attn_bwd_workspace(phsa_shape s, int topk);

/*
 * Stage (c) backward: gradients of the forward above with the selection held
 * fixed (a hard Top-K passes no gradient to Krepr, lambda or the scores).
 * With P_ij = exp(sm_scale q_i.k_j - lse_i), Delta_i = dO_i . O_i,
 * dS_ij = P_ij (dO_i . v_j - Delta_i):
 *   dV_j = sum_i P_ij dO_i;  dK_j = sm_scale sum_i dS_ij q_i;  dQ_i = sm_scale sum_j dS_ij k_j.
 * Sums run over every query head of the KV group. Deterministic: the same
 * inputs give bit-identical gradients.
 *   O, lse      the forward's outputs; dO bf16 [B, Hq, L, D] in
 *   workspace   device buffer of at least phsa_sparse_attn_bwd_workspace()
 *               bytes, owned by the caller, contents need not be initialised
 *   dQ          bf16 [B, Hq, L, D] out; dK, dV bf16 [B, Hkv, L, D] out
 */
int phsa_sparse_attn_bwd(const void* Q, const void* K, const void* V, const void* O,
                         const void* dO, const float* lse, const int32_t* block_idx,
                         const int32_t* block_cnt, phsa_shape s, int topk, float sm_scale,
                         void* workspace, size_t workspace_bytes, void* dQ, void* dK, void* dV,
                         void* stream);

/*
 * The backward pass above for callers that cannot allocate device memory (no
 * counterpart in the paper). Some callers may not call cudaMalloc where they
 * run the backward pass: engines that reserve all of HBM for their own pools
 * at start-up, plugin interfaces whose execute step must not allocate, or hot
 * loops that cannot afford cudaMalloc's implicit device synchronisation. This
 * entry point allocates nothing: its scratch is a fixed 64 MiB device array
 * inside the library, held by every GPU that loads the library until the
 * process exits. The caller still passes inputs and outputs, as for
 * phsa_sparse_attn_bwd, whose results it reproduces.
 *   - Shapes whose phsa_sparse_attn_bwd_workspace() exceeds 64 MiB return
 *     PHSA_ERR_WORKSPACE before any launch (for example B=1, Hq=16, Hkv=8,
 *     topk=8 fits up to L = 8192).
 *   - The first call on a device looks up the array's device address (with
 *     that device current) and caches it; make that first call before any
 *     stream capture begins.
 *   - All calls share the array and it keeps the last call's contents (each
 *     call clears what must start at zero). Calls that overlap on the GPU, for
 *     example on two streams, race on it: serialise them.
 */
int phsa_sparse_attn_bwd_noalloc(const void* Q, const void* K, const void* V, const void* O,
                                 const void* dO, const float* lse, const int32_t* block_idx,
                                 const int32_t* block_cnt, phsa_shape s, int topk, float sm_scale,
                                 void* dQ, void* dK, void* dV, void* stream);

/*
 * The whole path for tensors in HOST memory (no counterpart in the paper): one
 * training step of the attention -- stage (a), (b), the forward of (c) and its
 * backward pass for a given dO -- with the host<->device copies overlapped
 * with the kernels. Inputs Q, K, V, dO, punct_mask and outputs O, lse, dQ, dK,
 * dV, block_idx, block_cnt have the layouts of the calls above but are HOST
 * pointers; they should be page-locked (cudaHostAlloc / cudaHostRegister),
 * else the CUDA runtime stages the copies and they do not overlap. Any output
 * pointer may be NULL: that result is not copied back.
 *
 * Copies run on two streams the library owns (one per direction per device):
 * K and the mask are copied first, then Q, V and dO; stage (a) starts when K
 * has arrived, (b) when Q has, the forward when V has and the backward when
 * dO has. O, lse and the selection are copied back while the backward runs, dQ
 * while dK/dV are computed, dK and dV at the end. The kernels run on `stream`.
 *
 *   workspace   device buffer of at least phsa_step_host_workspace() bytes,
 *               256-byte aligned, owned by the caller: it holds the device
 *               copies of every input and output, the representative keys,
 *               the selection and the backward pass's scratch.
 *   done_event  NULL: `stream` is made to wait for the copies back, so that
 *               synchronising `stream` means the outputs are in host memory.
 *               Otherwise a cudaEvent_t (as void*) that the call records when
 *               the outputs are in host memory; `stream` then waits only for
 *               the kernels, and the next call's kernels can overlap this
 *               call's copies back.
 *
 * The copies in do not wait for earlier work on `stream`; they wait for the
 * previous call that used the same workspace to be done with it (copies back
 * included). A caller that alternates two workspaces therefore overlaps one
 * step's copies in with the previous step's kernels. The host buffers must
 * not be written (inputs) or read (outputs) until the call's work is done.
 * Validation as for the calls above; PHSA_ERR_WORKSPACE if the workspace is
 * NULL, misaligned or too small. Returns after enqueueing.
 */
size_t phsa_step_host_workspace(phsa_shape s, int topk);
int phsa_step_host(const void* Q, const void* K, const void* V, const void* dO,
                   const uint8_t* punct_mask, phsa_shape s, float lambda, phsa_select_params p,
                   void* O, float* lse, void* dQ, void* dK, void* dV, int32_t* block_idx,
                   int32_t* block_cnt, void* workspace, size_t workspace_bytes, void* done_event,
                   void* stream);
/* Waits for the last call on `workspace` and frees the library's events for
 * it; call before freeing a workspace that phsa_step_host used. */
int phsa_step_host_release(void* workspace);

/*
 * Decode: one new token per sequence, against per-sequence caches.
 * Layout: s.L is the cache capacity; K, V bf16 [B, Hkv, L, D]; punct_mask
 * uint8 [B, L]; Krepr bf16 [B, Hkv, floor(L/m), D]; seq_lens int32 [B] (device)
 * holds each sequence's token count, the new token included, so its query is
 * the token at p = seq_lens[b] - 1, with query block qb = floor(p/m). A length
 * of 0 means no query; a length < 0 or > L is a device-side error
 * (PHSA_ERR_DEVICE_INDEX) and that sequence is treated as empty.
 */

/*
 * Appends each sequence's new token to the caches: with p = seq_lens[b] - 1
 * (seq_lens counts the new token), K[b][g][p] = k_new[b][g] and
 * V[b][g][p] = v_new[b][g] for every KV head g, and punct_mask[b][p] =
 * flag_new[b] (nonzero = punctuation). A length <= 0 appends nothing; a length
 * > L is a device-side error (PHSA_ERR_DEVICE_INDEX) and appends nothing.
 *   k_new, v_new  bf16 [B, Hkv, D] in;  flag_new uint8 [B] in (may be NULL:
 *                 the mask is then left as it is)
 *   K, V          bf16 [B, Hkv, L, D] in/out;  punct_mask uint8 [B, L] in/out
 */
int phsa_decode_append(const void* k_new, const void* v_new, const uint8_t* flag_new,
                       const int32_t* seq_lens, phsa_shape s, void* K, void* V,
                       uint8_t* punct_mask, void* stream);

/*
 * Block-level caching of the representative keys (Section 3.2): for every
 * sequence whose length is a positive multiple of m, the block that the new
 * token has just filled, t = seq_lens[b]/m - 1, gets its representative key
 * (Eq. 6-8, the same arithmetic as phsa_build_block_repr); every other block
 * of Krepr is left as it is. Call after appending each token's K and mask;
 * build the initial Krepr of a prefilled cache with phsa_build_block_repr.
 */
int phsa_decode_update_repr(const void* K, const uint8_t* punct_mask, const int32_t* seq_lens,
                            phsa_shape s, float lambda, void* Krepr, void* stream);

/*
 * Selection for the new token (Eq. 8 / Algorithm 1 step 3 for one token):
 * the rule of phsa_select_blocks for a unit whose rows are the token p in
 * each of the G query heads of KV head g: forced F = {0..n_init-1} U
 * {qb-n_local+1..qb} clipped to [0, qb]; candidates are the full blocks
 * t <= qb-1 not in F; A[t] = sum over the G heads of softmax_t(sm_scale
 * q_h . Krepr[t]); min(topk-|F|, |C|) candidates by A descending, ties to
 * the lower t; ascending output, -1 padded.
 *   q         bf16 [B, Hq, D]       in (the new token of every sequence)
 *   block_idx int32 [B, Hkv, topk]  out; block_cnt int32 [B, Hkv] out
 */
int phsa_decode_select(const void* q, const void* Krepr, const int32_t* seq_lens, phsa_shape s,
                       phsa_select_params p, int32_t* block_idx, int32_t* block_cnt,
                       void* stream);

/*
 * Attention of the new token (Eq. 10-11 for row p): o = sum over keys j <= p
 * of the listed blocks of softmax_j(sm_scale q . k_j) v_j; lse its natural-log
 * log-sum-exp. Entries of block_idx must be -1 or 0 <= t <= qb, ascending;
 * others are skipped and recorded as PHSA_ERR_DEVICE_INDEX. A sequence with
 * no query gets o = 0 and lse = -inf.
 *   q    bf16 [B, Hq, D] in;  O bf16 [B, Hq, D] out;  lse fp32 [B, Hq] out
 */
int phsa_decode_attn(const void* q, const void* K, const void* V, const int32_t* block_idx,
                     const int32_t* block_cnt, const int32_t* seq_lens, phsa_shape s, int topk,
                     float sm_scale, void* O, float* lse, void* stream);

/*
 * One whole decode step in two launches: the selection of phsa_decode_select,
 * then the attention of phsa_decode_attn fused with phsa_decode_update_repr.
 * The block a sequence's new token has just filled is the query's own (local)
 * block: the attention reads it anyway and refreshes its representative key
 * from the copy in shared memory, and it is never a candidate of the same step,
 * so the selection does not depend on the refresh. Results are bit-identical
 * to the three calls update_repr, select, attn. Arguments as for those calls;
 * Krepr is read (candidates) and written (the filled blocks).
 */
int phsa_decode_step(const void* q, const void* K, const void* V, const uint8_t* punct_mask,
                     const int32_t* seq_lens, phsa_shape s, float lambda, phsa_select_params p,
                     void* Krepr, int32_t* block_idx, int32_t* block_cnt, void* O, float* lse,
                     void* stream);

/*
 * Prefill in chunks (block-level caching of Section 3.2; Eq. 3, 6, 7, 8;
 * Algorithm 1 step 2): appends a chunk of C = chunk_len tokens to every
 * sequence's caches and, from the same loads, computes the representative key
 * of every block of m = s.block_size tokens that the chunk completes, so a prefill does
 * not read K a second time for stage (a). With len = seq_lens[b] (the length
 * after the append, chunk included), the chunk takes positions
 * p = len - C + i, i in [0, C):
 *   K[b][g][p] = k_chunk[b][g][i], V[b][g][p] = v_chunk[b][g][i] for every
 *   KV head g, punct_mask[b][p] = flag_chunk[b][i] (when flag_chunk is given;
 *   otherwise the mask already holds the chunk's flags), and for every block t
 *   with len - C < (t + 1) m <= len, Krepr[b][g][t] = lambda M0 + (1 - lambda)
 *   Mp (Mp = M0 without punctuation), Eq. 6-8 over the block's m keys and
 *   flags, earlier ones read from the caches. The keys equal, bit for bit,
 *   those phsa_build_block_repr computes over the finished cache. Blocks the
 *   chunk leaves partial get no key yet.
 *   k_chunk, v_chunk bf16 [B, Hkv, C, D] in;  flag_chunk uint8 [B, C] in or NULL
 *   seq_lens int32 [B] in (device); s.L is the cache capacity
 *   K, V bf16 [B, Hkv, L, D], punct_mask uint8 [B, L], Krepr bf16
 *   [B, Hkv, floor(L/m), D]: in/out (device, caller-owned)
 * A length with len < C or len > L is a device-side error
 * (PHSA_ERR_DEVICE_INDEX) and that sequence is left untouched. chunk_len = 0
 * does nothing.
 */
int phsa_prefill_append(const void* k_chunk, const void* v_chunk, const uint8_t* flag_chunk,
                        const int32_t* seq_lens, int chunk_len, phsa_shape s, float lambda,
                        void* K, void* V, uint8_t* punct_mask, void* Krepr, void* stream);

/*
 * Synchronises `stream`, returns the device status word of the current
 * device (PHSA_OK or the first device-side error code recorded since the
 * last call) and clears it. Returns PHSA_ERR_CUDA if the synchronisation
 * itself fails.
 */
int phsa_get_device_status(void* stream);

/* Static, human-readable name of a phsa_status code. */
const char* phsa_status_string(int code);

/*
 * Optional per-kernel timing (no counterpart in the paper; an instrumentation
 * aid). phsa_profile_enable(1) makes every later kernel launch of the library
 * record a CUDA event before and after it on the launch stream; (0) stops it.
 * Returns the previous setting. phsa_profile_read waits for the recorded
 * events, fills up to max_kinds entries (static kernel names, total
 * milliseconds, launch counts; any pointer may be NULL) and clears the
 * records. Returns the number of kernel kinds, or PHSA_ERR_CUDA.
 */
int phsa_profile_enable(int on);
int phsa_profile_read(int max_kinds, const char** names, double* total_ms, int* launches);

/*
 * Diagnostic (no counterpart in the paper): runs the two tensor-core MMA
 * shapes of the forward kernel once on one CTA, S = A B^T and O = bf16(S) V,
 * with operands staged by TMA and accumulators in tensor memory, so that a
 * test can check the hardware path against a plain matrix product.
 *   A bf16 [128][128], B bf16 [64][128], V bf16 [64][128]  (device, in)
 *   S fp32 [128][64], O fp32 [128][128]                    (device, out)
 * Asynchronous on `stream`; a wait that times out is reported through
 * phsa_get_device_status as PHSA_ERR_TIMEOUT.
 */
int phsa_selftest_tcgen05(const void* A, const void* B, const void* V, float* S, float* O,
                          void* stream);

/*
 * Testing hook (no counterpart in the paper). With two query heads per KV
 * head, phsa_select_blocks runs the tensor-core selection at every block size
 * until, at block sizes 16 and 32, its per-query-block sums need more shared
 * memory than a switch point (227 KB by default: beyond about 64k tokens at
 * m = 16); longer sequences run on a warp-level MMA kernel. This call sets the
 * switch point to `bytes` (0, or more than 227 KB, restores the default) so
 * that a test can reach the warp-level pair kernels on short inputs; both
 * kernels compute the same selection. Returns the previous value. Affects
 * every later call in the process; not meant for production use.
 */
size_t phsa_test_set_select_tc_limit(size_t bytes);

/* Testing hook. The backward transposes the block lists (KV block -> the
 * query blocks that selected it) either in one launch, with one (batch, KV
 * head)'s bitmap of (KV span, query block) pairs in at most 160 KB of shared
 * memory, or in two launches through a bitmap in global memory. By default
 * the one-launch form runs at block size 64 while the bitmap fits (up to 1140
 * query blocks) and the two-launch form otherwise and at block sizes 16 and
 * 32. A nonzero `bytes` makes every block size take the one-launch form
 * while the bitmap fits in min(bytes, 160 KB), so that a test can reach
 * either form on short inputs; 0 restores the default. Both forms build the
 * same lists. Returns the previous setting (0: the default). Affects every
 * later call in the process; not meant for production use.
 */
size_t phsa_test_set_idx_smem_limit(size_t bytes);

/* Library version as "major.minor.patch". */
const char* phsa_version(void);

#ifdef __cplusplus
}
#endif

#endif /* PHSA_H */
