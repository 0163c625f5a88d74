// Kernel launchers behind the C ABI. Arguments are validated by the ABI layer
// (phsa_api.cu) before any of these run.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "phsa.h"

namespace phsa {

// Dynamic shared memory a CTA may use on sm_103a (227 KB); every kernel choice
// and every UNSUPPORTED check against it uses this one constant.
constexpr size_t kMaxDynSmem = 227u * 1024u;

// Kernel identities for the optional per-kernel timing (profile.cu).
enum KernelId {
    K_REPR = 0, K_SELECT, K_FWD, K_BWD_DELTA, K_BWD_MARK, K_BWD_BUILD, K_BWD_DKDV,
    K_BWD_DKDV_SUM, K_BWD_DQ, K_DEC_REPR, K_DEC_SELECT, K_DEC_ATTN, K_PREFILL_APPEND, K_COUNT
};
void prof_begin(int kid, cudaStream_t st);
void prof_end(int kid, cudaStream_t st);

// Brackets one kernel launch with the timing hooks.
struct ProfScope {
    int kid;
    cudaStream_t st;
    ProfScope(int k, cudaStream_t s) : kid(k), st(s) { prof_begin(kid, st); }
    ~ProfScope() { prof_end(kid, st); }
};

cudaError_t launch_block_repr(const void* K, const uint8_t* mask, const phsa_shape& s,
                              float lambda, void* Krepr, cudaStream_t st);

// Decode (one new token per sequence): repr of the block just filled, the
// selection and the attention of the newest token (decode.cu, block_repr.cu).
cudaError_t launch_decode_repr(const void* K, const uint8_t* mask, const int32_t* lens,
                               const phsa_shape& s, float lambda, void* Krepr, int* status,
                               cudaStream_t st);
size_t decode_select_smem_bytes(const phsa_shape& s, int topk);
cudaError_t launch_decode_select(const void* q, const void* Krepr, const int32_t* lens,
                                 const phsa_shape& s, const phsa_select_params& p, int32_t* idx,
                                 int32_t* cnt, int* status, cudaStream_t st);
cudaError_t launch_decode_attn(const void* q, const void* K, const void* V, const int32_t* idx,
                               const int32_t* cnt, const int32_t* lens, const phsa_shape& s,
                               int topk, float sm_scale, void* O, float* lse, int* status,
                               cudaStream_t st);
// The attention above, also refreshing the representative key of every block
// the new token has just filled (the work of launch_decode_repr).
cudaError_t launch_decode_attn_repr(const void* q, const void* K, const void* V,
                                    const int32_t* idx, const int32_t* cnt, const int32_t* lens,
                                    const phsa_shape& s, int topk, float sm_scale, void* O,
                                    float* lse, const uint8_t* mask, float lambda, void* Krepr,
                                    int* status, cudaStream_t st);
size_t decode_attn_smem_bytes(const phsa_shape& s, int topk);
// Writes the new token's k, v and punctuation flag at row len - 1 (decode.cu).
cudaError_t launch_decode_append(const void* k_new, const void* v_new, const uint8_t* flag,
                                 const int32_t* lens, const phsa_shape& s, void* K, void* V,
                                 uint8_t* mask, int* status, cudaStream_t st);
// Writes a chunk of C tokens (k, v, punctuation flags) at positions
// [len - C, len) of every sequence and the representative key of every block
// the chunk completes (prefill_append.cu).
cudaError_t launch_prefill_append(const void* k_chunk, const void* v_chunk, const uint8_t* flags,
                                  const int32_t* lens, int C, const phsa_shape& s, float lambda,
                                  void* K, void* V, uint8_t* mask, void* Krepr, int* status,
                                  cudaStream_t st);
// Punctuation indicator of token ids against a set of <= 4096 ids (punct.cu).
cudaError_t launch_punct_mask(const int32_t* ids, long long n, const int32_t* punct_ids,
                              int n_punct, uint8_t* mask, cudaStream_t st);

cudaError_t launch_select_tc(const void* Q, const void* Krepr, const phsa_shape& s,
                             const phsa_select_params& p, int32_t* idx, int32_t* cnt, int* status,
                             cudaStream_t st);
size_t select_tc_smem_bytes(const phsa_shape& s, int topk);
// The one-unit-per-step tcgen05 selection (select_tc_unit.cu), block size 64,
// which launch_select_tc runs for sequences of up to kSelectUnitMaxNqb query blocks.
constexpr int kSelectUnitMaxNqb = 1024;
cudaError_t launch_select_tc_unit(const void* Q, const void* Krepr, const phsa_shape& s,
                                  const phsa_select_params& p, int32_t* idx, int32_t* cnt,
                                  int* status, cudaStream_t st);
size_t select_tc_unit_smem_bytes(const phsa_shape& s, int topk);

cudaError_t launch_select_blocks(const void* Q, const void* Krepr, const phsa_shape& s,
                                 const phsa_select_params& p, int32_t* idx, int32_t* cnt,
                                 int* status, cudaStream_t st);

// tcgen05 forward for G = 2 at block sizes 64, 32, 16 (attn_fwd_tc.cu);
// launch_attn_fwd dispatches to it while its shared memory fits.
size_t attn_fwd_tc_smem_bytes(const phsa_shape& s, int topk);
cudaError_t launch_attn_fwd_tc(const void* Q, const void* K, const void* V, const int32_t* idx,
                               const int32_t* cnt, const phsa_shape& s, int topk, float sm_scale,
                               void* O, float* lse, int* status, cudaStream_t st);
cudaError_t launch_tc_selftest(const void* A, const void* B, const void* V, float* S, float* O,
                               int* status, cudaStream_t st);
bool make_tmap_bf16_rows128(CUtensorMap* map, const void* base, uint64_t rows, uint64_t planes,
                            uint32_t box_rows, uint32_t box_planes = 1);

cudaError_t launch_attn_fwd(const void* Q, const void* K, const void* V, const int32_t* idx,
                            const int32_t* cnt, const phsa_shape& s, int topk, float sm_scale,
                            void* O, float* lse, int* status, cudaStream_t st);

// Transposed selection, one entry per (b, kv head, KV block t): the offset and
// length of t's ascending list of selecting query blocks, its number of work
// chunks, and its first fp32 partial slot (-1 when it has a single chunk).
struct BwdTInfo {
    int off, n, nch, slot;
};
constexpr int kBwdChunk = 32;  // query blocks per dK/dV work item
// dK/dV work items are queued in two classes, items of at least 4 iterations
// first, then the shorter ones; inside a class each (b, g) holds one contiguous
// range, longest items first. A persistent kernel that takes the items in
// queue order keeps the Q/dO tiles of one or two (b, g) in L2 at a time and
// ends on short items, so the SMs finish together.
constexpr int kQueueClasses = 2;
constexpr int kShortItem = 4;
__host__ __device__ __forceinline__ int queue_class(int n_it) {
    return n_it >= kShortItem ? 0 : 1;
}

// tcgen05 backward kernels for G = 2 (attn_bwd_tc.cu).
struct BwdLayout;
cudaError_t launch_dkdv_tc(const void* Q, const void* K, const void* V, const void* dO,
                           const float* lse, const float* delta, const BwdTInfo* tinfo,
                           const int32_t* qlist, const uint8_t* masks, const int2* queue,
                           int* qctl, const phsa_shape& s, int topk, const BwdLayout& l,
                           float sm_scale, void* dK, void* dV, float* partial, int* arrive,
                           int* status, cudaStream_t st);
// Whether dq_tc_kernel's shared memory (tiles + the block list) fits for topk
// at block size m.
bool dq_tc_fits(int topk, int block_size = 64);
// dQ (and Delta). At m < 64 the span lists are ulist/ucnt/umask (the unions
// of the span's query-block lists); at m = 64, idx/cnt.
cudaError_t launch_dq_tc(const void* Q, const void* K, const void* V, const void* O,
                         const void* dO, const float* lse, float* delta, const int32_t* idx,
                         const int32_t* cnt, const int32_t* ulist, const int32_t* ucnt,
                         const uint8_t* umask, const phsa_shape& s, int topk, float sm_scale,
                         void* dQ, int* status, cudaStream_t st);

// Backward workspace layout (all offsets 256-byte aligned). The transposed
// selection has one row per KV span of 64 keys and one column per query block
// of m tokens (at m = 64 a span is a block); at m < 64 a mask row per span
// records which of its kSub blocks each query block selected, and the dQ pass
// reads the union of each span's query-block lists (ucnt, ulist, umask).
struct BwdLayout {
    // qctl: item counts of the kQueueClasses queue classes, then the ticket
    // counter of the persistent dK/dV kernel (zeroed with the bitmap by one memset)
    size_t qctl, bits, masks, tinfo, qlist, work, nwork, queue, delta, partial, arrive, ucnt, ulist,
        umask, total;
    int nqb;    // query blocks of m tokens
    int nrows;  // KV spans of 64 keys
    int kSub, words, mrow, chunk, work_max, slot_max, ucap;
};
BwdLayout bwd_layout(const phsa_shape& s, int topk);

// after_dq (optional) is recorded on st once dQ is complete, before dK/dV
// finish, so that a caller can start copying dQ out early.
cudaError_t launch_attn_bwd(const void* Q, const void* K, const void* V, const void* O,
                            const void* dO, const float* lse, const int32_t* idx,
                            const int32_t* cnt, const phsa_shape& s, int topk, float sm_scale,
                            void* ws, void* dQ, void* dK, void* dV, int* status,
                            cudaStream_t st, cudaEvent_t after_dq = nullptr);

// The status word of the current device (phsa_api.cu); null if it cannot be found.
int* device_status_word();
// PHSA_OK for cudaSuccess, PHSA_ERR_CUDA otherwise (the mapping of every entry point).
int status_of(cudaError_t e);
// Shape and budget checks of the C ABI (phsa_api.cu): PHSA_OK or an error code.
int validate_shape(const phsa_shape& s);
// The backward's shape and budget checks (block sizes 16 and 32 for GQA pairs).
int validate_bwd(const phsa_shape& s, int topk);
int validate_topk(const phsa_shape& s, int topk);
// Shared-memory bytes of the selection kernel for this shape and budget.
size_t select_smem_bytes(const phsa_shape& s, int topk);
// Whether a GQA-pair selection runs on the tcgen05 kernel (select_tc.cu): always
// at m = 64; at m = 16 and 32 while its per-query-block sums fit under the
// switch point (kMaxDynSmem, lowered only by phsa_test_set_select_tc_limit).
bool select_uses_tc(const phsa_shape& s, int topk);

}  // namespace phsa
