/*
 * spire.h -- C ABI of libspire: the KV-cache-bound attention of one SPIRe
 * speculation round (Neelam et al., "SPIRe: Boosting LLM Inference Throughput
 * with Speculative Decoding", arXiv 2504.06419), on one NVIDIA GB300 (sm_103a).
 *
 * A speculation round is k draft-model passes followed by one target-model
 * pass over the k+1 block tokens in parallel (Section 2, the Throughput
 * Multiplier equation and the definitions of t_draft / t_verify beneath it;
 * Fig. 1 caption).  In the large-batch long-context regime the cost of both is
 * loading the KV cache (Section 1; Section 3.1).  This library implements that
 * part:
 *
 *   spire_verify_attention        the target's verification attention: k+1
 *                                 causal block queries per sequence over its
 *                                 full, paged, ragged bf16 KV cache, with GQA.
 *   spire_draft_sparse_attention  the draft's StreamingLLM attention: sink
 *                                 entries plus a sliding window of feedback-
 *                                 memory entries m_{<t} (Sections 3.1, 3.3),
 *                                 over a bounded cache.
 *   spire_feedback_append         the draft step's cache update: mix the
 *                                 token's activations into each layer's memory
 *                                 vector, project it to K/V and store it in
 *                                 the bounded cache (Section 3.3).
 *   spire_magicdec_attention      the MagicDec baseline's draft attention:
 *                                 sink + window over the target's own paged
 *                                 cache, positions inside that reduced cache.
 *   spire_verify_tokens           the round's token verification: modified
 *                                 rejection sampling of the draft tokens
 *                                 (Section 1).
 *
 * Conventions common to every call
 *   - All tensor arguments are DEVICE pointers, owned by the caller; the
 *     library keeps no pointer after a call returns and allocates nothing.
 *     One exception: `out` of spire_verify_attention(_noalloc),
 *     spire_draft_sparse_attention and spire_magicdec_attention may also be
 *     pinned host memory mapped into the device's address space
 *     (cudaHostAlloc / cudaHostRegister memory on a system with unified
 *     addressing, where the host pointer is valid on the device).  Those
 *     kernels only store to `out`, with plain stores, so the results reach
 *     the host without a separate copy (zero-copy; over NVLink-C2C on a
 *     Grace host) and are visible there once the stream has reached the end
 *     of the call.
 *   - Every call is asynchronous on `stream` (a cudaStream_t passed as void*;
 *     NULL is the legacy default stream).  Only spire_get_device_error and
 *     spire_get_cta_times synchronise.
 *   - Arguments that can be checked on the host are checked before anything is
 *     launched; a failing check returns a status and launches nothing.
 *   - Values that live on the device (ctx_lens, block_table) are checked by
 *     the kernels.  A sequence whose values break the rules gets NaN in every
 *     one of its output rows, and a bit is set in the device error word in the
 *     workspace (read it with spire_get_device_error).  No kernel traps, reads
 *     out of bounds or waits without a time limit.
 *   - Results are deterministic: the split of the KV range across SMs depends
 *     only on ctx_lens and the shapes, and the splits are merged in a fixed
 *     order, so repeated calls give bit-identical outputs.
 *   - Pointers to q, caches and out must be 16-byte aligned, the workspace
 *     256-byte aligned.
 */
#ifndef SPIRE_H
#define SPIRE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define SPIRE_API __attribute__((visibility("default")))
#else
#define SPIRE_API
#endif

/* Status of a host call. */
typedef enum spire_status {
    SPIRE_OK = 0,
    SPIRE_ERR_INVALID_ARG = 1,  /* null pointer, bad shape, misalignment, ... */
    SPIRE_ERR_UNSUPPORTED = 2,  /* valid but not implemented (head_dim, rows) */
    SPIRE_ERR_WORKSPACE = 3,    /* workspace missing or smaller than required */
    SPIRE_ERR_CUDA = 4          /* a CUDA runtime/driver call failed */
} spire_status;

/* Bits of the device error word (spire_get_device_error). */
#define SPIRE_DEVERR_CTX_LEN 1u  /* a ctx_lens entry outside its allowed range */
#define SPIRE_DEVERR_PAGE_ID 2u  /* a block_table entry outside [0, num_pages) */
#define SPIRE_DEVERR_TIMEOUT 4u  /* a bounded wait inside a kernel gave up */
#define SPIRE_DEVERR_VALUE 8u    /* an input value outside its domain (spire_verify_tokens) */

/* Shapes shared by both kernels. */
typedef struct spire_attn_desc {
    int32_t batch;             /* B >= 0 sequences (B == 0: nothing to do) */
    int32_t num_q_heads;       /* Hq >= 1 */
    int32_t num_kv_heads;      /* Hkv >= 1, Hq % Hkv == 0; query head h reads
                                  KV head h / (Hq / Hkv) (grouped-query) */
    int32_t head_dim;          /* D, 64 or 128 */
    int32_t page_size;         /* verify: tokens per KV page, must be 64 */
    int32_t max_pages_per_seq; /* verify: columns of block_table */
    int32_t num_pages;         /* verify: pages held by k_cache / v_cache */
    float softmax_scale;       /* score = softmax_scale * <q, k>; finite, > 0
                                  (1.0 when q is pre-scaled by 1/sqrt(D)) */
} spire_attn_desc;

/* Largest number of query rows one KV head serves: (Hq/Hkv) * (k+1) <= 128. */
#define SPIRE_MAX_ROWS_PER_KV_HEAD 128

/*
 * spire_verify_workspace_bytes -- workspace size for spire_verify_attention.
 * Depends only on the shapes (batch, heads, head_dim) and k, not on the
 * device or on ctx_lens.  Returns 0 if desc is NULL or k < 0.
 */
SPIRE_API size_t spire_verify_workspace_bytes(const spire_attn_desc *desc, int32_t k);

/*
 * spire_verify_attention -- verification attention of one speculation round
 * (Section 2: t_verify is a target pass over the k+1 block tokens in
 * parallel; Table 1 caption: a round yields 1..k+1 tokens).
 *
 *   q            bf16 [B, k+1, Hq, D]; block row i of sequence b.
 *   k_cache      bf16 [num_pages, Hkv, page_size, D]; key of token j of
 *                sequence b, KV head g, is
 *                k_cache[block_table[b][j / page_size], g, j % page_size, :].
 *   v_cache      bf16, same layout as k_cache.
 *   block_table  int32 [B, max_pages_per_seq]; only the first
 *                ceil(ctx_lens[b] / page_size) entries of row b are read, and
 *                each must lie in [0, num_pages).
 *   ctx_lens     int32 [B] on the device: L_b, the number of cache entries of
 *                sequence b INCLUDING the k+1 block tokens, whose K/V the
 *                caller has already written.  Must satisfy
 *                k+1 <= L_b <= max_pages_per_seq * page_size.
 *   k            speculation depth, k >= 0.
 *   out          fp32 [B, k+1, Hq, D]:
 *                out[b,i,h] = sum_j softmax_j(scale * <q[b,i,h], K_j>) V_j
 *                over keys j < L_b - k + i (row i is causal within the block:
 *                it equals single-query decoding at length L_b - k + i).
 *   workspace    device buffer of >= spire_verify_workspace_bytes(desc, k)
 *                bytes; holds the split plan, split partials and the device
 *                error word.  Contents need no initialisation.  Calls that
 *                share a workspace must be ordered (same stream).
 * Returns SPIRE_OK once the work is enqueued.
 */
SPIRE_API spire_status spire_verify_attention(const void *q, const void *k_cache,
                                    const void *v_cache,
                                    const int32_t *block_table,
                                    const int32_t *ctx_lens, int32_t k,
                                    const spire_attn_desc *desc, float *out,
                                    void *workspace, size_t ws_bytes,
                                    void *stream);

/*
 * spire_verify_attention_noalloc -- spire_verify_attention for callers that
 * cannot allocate device memory at call time (for example a serving engine
 * that gives all free GPU memory to its KV-cache pool at start-up, or a
 * plugin host that passes only input and output pointers).  The paper has no
 * counterpart: this is a property of the library, not of the method.
 *
 * Arguments and results are those of spire_verify_attention without the
 * workspace: its scratch (split partials, arrival counters, error words) is
 * one file-scope device array of 32 MiB, reserved on every GPU that loads
 * libspire until the process exits.  Nothing is allocated by the call.
 *   - A valid, non-empty shape whose workspace (spire_verify_workspace_bytes)
 *     exceeds 32 MiB returns SPIRE_ERR_WORKSPACE; at head_dim 128 that allows
 *     up to about 60 query rows per KV head ((Hq/Hkv)*(k+1)).  Every other
 *     case returns what spire_verify_attention returns: an empty batch is a
 *     no-op (SPIRE_OK), an unsupported page size SPIRE_ERR_UNSUPPORTED, null
 *     or misaligned pointers SPIRE_ERR_INVALID_ARG.
 *   - The first call on a device looks up the array's device address
 *     (cudaGetSymbolAddress) with that device current; make that first call
 *     before any stream capture.  The address is looked up again when the
 *     device's context has changed since (after cudaDeviceReset, for
 *     example), so such a call, too, belongs outside a capture.
 *   - All calls share the one array: calls that may overlap on the GPU (on
 *     different streams, or from different threads) race and must not be
 *     issued.  The array keeps the last call's contents; each call clears what
 *     must start at zero.  spire_get_device_error and spire_get_cta_times are
 *     not available for it.
 */
SPIRE_API spire_status spire_verify_attention_noalloc(const void *q, const void *k_cache,
                                                      const void *v_cache,
                                                      const int32_t *block_table,
                                                      const int32_t *ctx_lens, int32_t k,
                                                      const spire_attn_desc *desc, float *out,
                                                      void *stream);

/*
 * spire_draft_workspace_bytes -- workspace size for
 * spire_draft_sparse_attention.  Returns 0 for invalid arguments.
 */
SPIRE_API size_t spire_draft_workspace_bytes(const spire_attn_desc *desc, int32_t n_sink,
                                   int32_t window);

/*
 * spire_draft_sparse_attention -- one draft-model attention step with the
 * StreamingLLM mask (Section 3.1: attention sink plus sliding window, a KV
 * cache of constant size; Section 4: window 64, sink 1 in the paper) over
 * feedback-memory entries (Section 3.3: z_t = Attention(x_t, m_{<t}); each
 * draft layer keeps its own memory m^i, so each layer has its own cache).
 *
 *   q         bf16 [B, Hq, D]: one query per sequence.
 *   kv        bf16 [B, 2, Hkv, S, D], S = n_sink + window; index 0 holds K,
 *             1 holds V.  Memory entry p lives in slot spire_draft_slot(p):
 *             sinks p < n_sink are fixed, later entries form a ring.
 *   ctx_lens  int32 [B] on the device: t_b >= 1, the number of memory entries
 *             m_0..m_{t-1} written so far.  The query sees
 *             V(t) = {p < min(n_sink, t)} u {max(0, t - window) <= p < t},
 *             which occupy exactly slots [0, min(t, S)).  The current token's
 *             own entry is not visible (m_{<t}); pass t+1 after writing it for
 *             self-inclusive StreamingLLM attention.
 *   n_sink    >= 0 sink entries;  window >= 1 window entries.
 *   out       fp32 [B, Hq, D].
 *   workspace >= spire_draft_workspace_bytes(desc, n_sink, window) bytes.
 * desc->page_size / max_pages_per_seq / num_pages are ignored.
 */
SPIRE_API spire_status spire_draft_sparse_attention(const void *q, const void *kv,
                                          const int32_t *ctx_lens,
                                          int32_t n_sink, int32_t window,
                                          const spire_attn_desc *desc,
                                          float *out, void *workspace,
                                          size_t ws_bytes, void *stream);

/*
 * Draft-step cache update: the feedback-memory append.
 *
 * After the draft model has run token t, each of its layers i gets a new
 * memory vector m_t^i, the softmax(w_i)-weighted average of the token's
 * activations x_t^0 (embedding) .. x_t^{n_layer} (Section 3.3, the per-layer
 * memory equation; layers share neither memory vectors nor projections).
 * Layer i attends to keys and values of its memory entries, so the vector is
 * projected by the layer's key and value matrices and stored in slot
 * spire_draft_slot(p) of the layer's bounded cache (Section 3.1), where p is
 * the number of entries before it.  The paper names no positional scheme,
 * only that SPIRe uses the token's original-text position (Section 3.1,
 * footnote); with rope_theta > 0 keys are turned by that position (rotary,
 * half-split pairs (d, d + D/2), angle p * rope_theta^(-2d/D)).
 */
typedef struct spire_append_desc {
    int32_t batch;            /* B >= 0 sequences, one new entry each (0: nothing to do) */
    int32_t num_act;          /* n_layer + 1 activations mixed (1..16), x^0 = embedding */
    int32_t num_draft_layers; /* n_dl (1..16): memory vector, projection and cache per layer */
    int32_t d_model;          /* activation width, a multiple of 64 (64..65536) */
    int32_t num_kv_heads;     /* Hkv >= 1 */
    int32_t head_dim;         /* D: 64 or 128 */
    int32_t n_sink;           /* >= 0 sink slots of each cache */
    int32_t window;           /* >= 1 window slots of each cache */
    float rope_theta;         /* > 0: rotate keys by position; 0: no rotation */
} spire_append_desc;

/*
 * spire_feedback_append_workspace_bytes -- workspace size for
 * spire_feedback_append (the device error words; the same 2304 bytes for
 * every valid descriptor).  Returns 0 for invalid arguments.
 */
SPIRE_API size_t spire_feedback_append_workspace_bytes(const spire_append_desc *desc);

/*
 * spire_feedback_append -- write one memory entry per sequence into every
 * draft layer's bounded cache:
 *     m[i, b]      = sum_l softmax(mix_w[i, :])_l * x[l, b, :]
 *     K[i, b, g, :] = w_kv[i, g*D .. g*D + D - 1, :]               . m[i, b]
 *     V[i, b, g, :] = w_kv[i, Hkv*D + g*D .. Hkv*D + g*D + D - 1, :] . m[i, b]
 * K rotated by pos[b] when rope_theta > 0, both rounded to nearest-even bf16
 * and stored at kv[i, b, 0 (K) / 1 (V), g, spire_draft_slot(pos[b]), :].
 *
 *   x        bf16 [num_act, B, d_model]: the token's activations.
 *   mix_w    fp32 [n_dl, num_act]: the learnable weights w_{il}, un-normalised.
 *   w_kv     bf16 [n_dl, 2*Hkv*D, d_model]: per layer the key rows, then the
 *            value rows (row-major, d_model contiguous).
 *   pos      int32 [B] on the device: p >= 0, the entry's logical position.
 *   kv       bf16 [n_dl, B, 2, Hkv, n_sink + window, D]: the caches (layer i's
 *            cache is the [B, 2, Hkv, S, D] block spire_draft_sparse_attention
 *            reads), updated in place; no other slot is written.
 *   workspace >= spire_feedback_append_workspace_bytes(desc) bytes.
 * The projection is linear, so the kernel computes sum_l a_l (W x_l) with
 * a = softmax(mix_w[i, :]): exact bf16 products accumulated in fp32 on the
 * tensor cores, the accumulators mixed in fp32; an entry is within one bf16
 * unit of the exactly rounded value up to the fp32 accumulation error.  One
 * launch (thread-block clusters, programmatic dependent launch; a one-thread
 * error-word clear before it only for grids above 512 CTAs).  A sequence with
 * pos[b] < 0 is not written and sets SPIRE_DEVERR_CTX_LEN.  Pointers x, w_kv
 * and kv must be 16-byte aligned, the workspace 256-byte aligned.
 */
SPIRE_API spire_status spire_feedback_append(const void *x, const float *mix_w,
                                             const void *w_kv, const int32_t *pos,
                                             const spire_append_desc *desc, void *kv,
                                             void *workspace, size_t ws_bytes,
                                             void *stream);

/*
 * MagicDec draft attention -- the paper's main baseline (Section 4): the
 * target model drafts for itself, attending with a StreamingLLM mask (sink
 * entries plus a sliding window; sink 1, window 64 in the paper) to its own
 * paged KV cache, and, like StreamingLLM, gives entries their positions inside
 * that reduced cache rather than in the text (Section 3.1, footnote).
 *
 * For sequence b with t = ctx_lens[b] visible cache entries (the current
 * token's own included), the visible positions are [0, s) and [w0, t) with
 * s = min(n_sink, t), w0 = max(s, t - window); entry p gets cache index c = p
 * (sinks) or s + (p - w0) (window), and the query the last index, n - 1, with
 * n the number of visible entries.  The target cache holds keys turned by
 * their text position (rotary, half-split pairs (d, d + D/2), angle
 * p * rope_theta^(-2d/D)); each visible key is turned by (c - p) and the
 * query (given unrotated) by n - 1, both rounded to bf16, values unchanged;
 * then softmax attention as spire_draft_sparse_attention.  rope_theta = 0
 * skips every rotation.
 *
 *   q          bf16 [B, Hq, D], not rotated.
 *   k_cache, v_cache, block_table: the target's paged cache as for
 *              spire_verify_attention.
 *   ctx_lens   int32 [B] on the device: 1 <= t <= max_pages_per_seq * 64.
 *   n_sink >= 0, window >= 1, n_sink + window <= 65536.
 *   out        fp32 [B, Hq, D].
 *   workspace  >= spire_magicdec_workspace_bytes(desc, n_sink, window) bytes:
 *              the reduced cache, the turned queries and the attention's own
 *              workspace.
 * A length out of range, or a block-table entry outside the cache among the
 * visible entries, gives NaN rows and sets SPIRE_DEVERR_CTX_LEN.
 */
SPIRE_API size_t spire_magicdec_workspace_bytes(const spire_attn_desc *desc, int32_t n_sink,
                                                int32_t window);

SPIRE_API spire_status spire_magicdec_attention(const void *q, const void *k_cache,
                                                const void *v_cache,
                                                const int32_t *block_table,
                                                const int32_t *ctx_lens, int32_t n_sink,
                                                int32_t window, float rope_theta,
                                                const spire_attn_desc *desc, float *out,
                                                void *workspace, size_t ws_bytes,
                                                void *stream);

/*
 * Token verification of a speculation round (modified rejection sampling).
 *
 * Every emitted token is a sample of the target's own distribution (Section
 * 1; the token verification algorithm of the paper's experiments, Section 6).
 * For sequence b with draft tokens x_1..x_k drawn from the draft
 * distributions q_1..q_k and target distributions p_1..p_{k+1} from the
 * verification pass:
 *   - draft i is accepted with probability min(1, p_i(x_i) / q_i(x_i)): with a
 *     uniform u_i in [0, 1), accepted iff u_i * q_i(x_i) < p_i(x_i) (binary32);
 *     j is the number of leading accepted drafts;
 *   - the round then draws one token: from max(0, p_{j+1} - q_{j+1})
 *     normalised when j < k (from p_{j+1} if that residual has no positive
 *     entry), from p_{k+1} when j = k.  A draw from weights w is the
 *     exponential race argmax_v w_v / E_v over w_v > 0 (binary32 quotient, ties
 *     to the smallest v) with E_v ~ Exp(1) supplied by the caller, which picks
 *     v with probability w_v / sum(w).
 * Random numbers are inputs, so a call is deterministic.
 */

/*
 * spire_verify_tokens_workspace_bytes -- workspace size for
 * spire_verify_tokens (one partial per sequence and 4096-entry vocabulary
 * chunk, and the device error word).  Returns 0 for invalid shapes.
 */
SPIRE_API size_t spire_verify_tokens_workspace_bytes(int32_t batch, int32_t k, int32_t vocab);

/*
 * spire_verify_tokens --
 *   p            fp32 [B, k+1, V]: target distributions p_1..p_{k+1}.
 *   q            fp32 [B, k, V]:   draft distributions q_1..q_k (may be NULL if k = 0).
 *   draft_tokens int32 [B, k]:     x_1..x_k (may be NULL if k = 0).
 *   u            fp32 [B, k]:      acceptance uniforms in [0, 1) (may be NULL if k = 0).
 *   e            fp32 [B, V]:      Exp(1) variates for the round's one draw.
 *   batch 0..65535 (0: nothing to do, any pointer may be NULL), k 0..31, vocab V >= 1.
 *   out_tokens   int32 [B, k+1]:   x_1..x_j, the drawn token, then -1.
 *   n_accepted   int32 [B]:        j.
 * Only the rows the round needs are read (p_{j+1}, q_{j+1}, E and k gathered
 * entries).  A draft token outside [0, V) counts as rejected and sets
 * SPIRE_DEVERR_CTX_LEN; an E value that is not > 0 is skipped, and a draw with
 * no candidate yields -1; both set SPIRE_DEVERR_VALUE.  Pointers must be
 * 4-byte aligned (p, q and e 16-byte aligned when V is a multiple of 4), the
 * workspace 256-byte aligned.
 */
SPIRE_API spire_status spire_verify_tokens(const float *p, const float *q,
                                           const int32_t *draft_tokens, const float *u,
                                           const float *e, int32_t batch, int32_t k,
                                           int32_t vocab, int32_t *out_tokens,
                                           int32_t *n_accepted, void *workspace,
                                           size_t ws_bytes, void *stream);

/*
 * spire_test_stall_next_call -- a test hook for the failure path; the paper
 * has no counterpart, and production code does not call it.  In the next
 * spire_verify_attention or spire_draft_sparse_attention call made by the
 * calling host thread, the producer of every CTA that reaches pair `pair`
 * (= b * num_kv_heads + g) issues no loads from that pair on, so no copy of
 * it is ever in flight and the bounded waits for it run out (2 s).  The call
 * returns normally; its kernels give up, record SPIRE_DEVERR_TIMEOUT in the
 * device error word (spire_get_device_error), leave the affected outputs
 * unspecified, drain their own copies and tensor-core work, free tensor
 * memory, and leave the context usable.  The stalling kernels are separate
 * test instantiations (head_dim 128 only; at other head dims the call runs
 * normally), so the production kernels carry no trace of the hook.  Returns
 * SPIRE_ERR_INVALID_ARG for pair < 0 (nothing is armed then).
 */
SPIRE_API spire_status spire_test_stall_next_call(int32_t pair);

/*
 * spire_stream_read -- a measurement helper; the paper has no counterpart.
 * One kernel launch that reads `bytes` of device memory at `src` once and
 * computes nothing: one CTA per SM streams a contiguous run of 16 KB chunks
 * through a ring of shared-memory stages with bulk async copies, as the
 * attention kernels stream their K/V tiles.  Its time is the floor of any
 * single launch of this library that must read that many bytes (launch,
 * first-byte latency and the stream), against which calls that move tens of
 * MB -- a draft step, the feedback append, token verification -- are
 * compared.  src must be 16-byte aligned and bytes a multiple of 16
 * (SPIRE_ERR_INVALID_ARG otherwise); bytes = 0 is a no-op.  Nothing is
 * written; asynchronous on `stream`.
 */
SPIRE_API spire_status spire_stream_read(const void *src, size_t bytes, void *stream);

/*
 * spire_draft_slot -- slot of logical memory position p >= 0 in the bounded
 * draft cache (Section 3.1: attention sinks kept, a sliding window over the
 * rest, so the cache never grows): p if p < n_sink, else
 * n_sink + (p - n_sink) mod window.  Returns -1 for p < 0, n_sink < 0 or
 * window < 1.  Exported host function (for callers through an FFI).
 *
 * spire_draft_slot_inline is the same function, defined here for host code
 * and for CUDA device code (compiled by nvcc it is __host__ __device__).  It
 * is the one definition: the exported function and the kernel that writes
 * new entries into the cache (spire_feedback_append) both use it.
 */
#if defined(__CUDACC__)
#define SPIRE_HOST_DEVICE __host__ __device__
#else
#define SPIRE_HOST_DEVICE
#endif
static inline SPIRE_HOST_DEVICE int64_t spire_draft_slot_inline(int64_t pos, int32_t n_sink,
                                                               int32_t window) {
    if (pos < 0 || n_sink < 0 || window < 1) return -1;
    if (pos < n_sink) return pos;
    return n_sink + (pos - n_sink) % window;
}

SPIRE_API int64_t spire_draft_slot(int64_t pos, int32_t n_sink, int32_t window);

/*
 * spire_test_draft_slots -- a test hook; the paper has no counterpart.  One
 * kernel launch that writes spire_draft_slot_inline(p, n_sink, window),
 * evaluated on the device, to out[p] for p = 0 .. n-1 (int64, device memory,
 * 8-byte aligned), so that tests can hold the device evaluation of the inline
 * helper (the one the cache-writing kernel uses) against the host's.
 * Asynchronous on `stream`.  Returns SPIRE_ERR_INVALID_ARG for n < 0 or a null
 * or misaligned out (n = 0 is a no-op).
 */
SPIRE_API spire_status spire_test_draft_slots(int64_t *out, int64_t n, int32_t n_sink,
                                              int32_t window, void *stream);

/*
 * spire_get_device_error -- copy the device error word of the most recent
 * call that used `workspace` into *code_out (0 = no error, else an OR of
 * SPIRE_DEVERR_* bits).  Synchronises `stream`.
 */
SPIRE_API spire_status spire_get_device_error(const void *workspace, int32_t *code_out,
                                    void *stream);

/*
 * spire_get_cta_times -- the per-CTA timing record of the most recent
 * spire_verify_attention or spire_draft_sparse_attention call that used
 * `workspace` (ws_bytes of it): for each of the call's n CTAs (one per SM, in
 * CTA order) two %globaltimer readings in nanoseconds, when the CTA started
 * its first tile (after the launch dependency) and when it finished its last
 * output or merge.  The difference is that SM's busy time; the split of the
 * KV range gives every CTA the same number of tiles (within one), so the
 * spread shows how evenly the time follows.  Synchronises `stream`, writes n
 * to *n_out and the first min(n, max_ctas) pairs to ns_out[2i], ns_out[2i+1]
 * (host memory).  Returns SPIRE_ERR_WORKSPACE if ws_bytes cannot hold the
 * record of n CTAs.  The record is meaningless after any other call on the
 * same workspace (which does not write it).
 */
SPIRE_API spire_status spire_get_cta_times(const void *workspace, size_t ws_bytes,
                                 uint64_t *ns_out, int32_t max_ctas, int32_t *n_out,
                                 void *stream);

/* spire_status_string -- static, human-readable name of a status. */
SPIRE_API const char *spire_status_string(spire_status status);

#ifdef __cplusplus
}
#endif

#endif /* SPIRE_H */
