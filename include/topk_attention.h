/*
 * topk_attention.h -- C ABI of libtopk.so: top-k attention and the top-k
 * feed-forward layer (Gupta et al., "Memory-efficient Transformers via Top-k
 * Attention", arXiv 2106.06899) on NVIDIA GB300 (sm_103a).
 *
 * Operations
 *   topk_attn_fwd  -- Eq. 4 (Sec. 2.2):  out = softmax(top-k(Q K^T)) V, row by
 *                     row, the softmax taken over the k kept entries only.
 *                     The temperature of Eq. 1 is folded into Q by the caller
 *                     (footnote to Eq. 1).  Optional causal mask, Eq. 2: the
 *                     queries are the last Lq of the Lk positions (Lq <= Lk;
 *                     Lq < Lk is decoding against a key/value cache), and key
 *                     j is valid for query i iff j <= i + Lk - Lq.
 *   topk_attn_fwd_masked -- the same under Eq. 2's general mask B in {0, -inf}:
 *                     per-batch key counts and an arbitrary bit mask as well.
 *   topk_ffn_fwd   -- Eq. 3 with top-k (Sec. 2.1 "Feed-forward as attention"):
 *                     out = sum over the k largest s_j = x . W1_j of
 *                     ReLU(s_j) * W2_j.  Keys and values are the ROWS of W1
 *                     and W2.
 *   topk_attn_bwd  -- the backward pass of Eq. 4 for the kept set the forward
 *   topk_ffn_bwd      pass cached (Sec. 2.2 "Improving efficiency through
 *                     top-k attention"): gradients of q, k, v (x, W1, W2)
 *                     from dout, the kept indices and their scores, with the
 *                     activation recomputed from the cached scores.
 * Query chunking (Sec. 2.2 "Query chunking") bounds scheduling only: results
 * never depend on `chunk`, and no [chunk x L_K] score matrix is ever stored
 * in device memory.
 *
 * Selection rule: each row keeps the first k entries of the total order
 * (score descending, key index ascending) among its valid keys, i.e. ties go
 * to the lower key index.  A row with fewer than k valid keys keeps all of
 * them; a row with none outputs zeros (its indices are all -1).
 *
 * Conventions shared by every call
 *   - Tensor pointers are DEVICE pointers (except the *_host entry points),
 *     owned by the caller, contiguous, row-major, 16-byte aligned.
 *   - Shapes: q, out [B, H, Lq, d]; k, v [B, H, Lk, d];
 *             x [N, d_model]; W1, W2 [d_ff, d_model]; ffn out [N, d_model].
 *   - dtype: TOPK_F32 (fp32 in/out, fp32 FMA scores, never TF32) or
 *            TOPK_BF16 (bf16 in/out, fp32 accumulation).  The feed-forward
 *            call takes bf16 inputs and writes fp32 output.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream).  Calls
 *     enqueue work and return without synchronising.
 *   - Every argument is validated before anything is launched, so an error
 *     return never leaves a partial write.
 *   - Scratch, where a call needs it, is taken on `stream` from a
 *     stream-ordered memory pool that the library owns (one per device) and
 *     returned to it on `stream`; its size is reported by the
 *     *_workspace_bytes queries and is never proportional to Lq * Lk: a
 *     fixed amount per SM for attention (plus, when a grid of few query
 *     tiles is split into key parts, each part's kept list per row), linear
 *     in the tokens for the feed-forward layer and in the cache for the
 *     backward calls.  The pool keeps returned memory
 *     reserved for later calls (up to the largest amount in use at once),
 *     so that repeated calls do not map device memory again each time, until
 *     topk_pool_trim() hands it back or the process exits;
 *     topk_pool_usage() reports it.
 *
 * Return codes: 0 on success, else one of the negative TOPK_ERR_* values;
 * topk_error_string() describes them.
 */
#ifndef TOPK_ATTENTION_H
#define TOPK_ATTENTION_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum { TOPK_F32 = 0, TOPK_BF16 = 1 } topk_dtype;

enum {
  TOPK_OK = 0,
  TOPK_ERR_INVALID_ARG = -1, /* null pointer, non-positive size, topk < 1 or > keys, chunk < 1,
                                causal with Lq > Lk, negative mask stride, unknown dtype */
  TOPK_ERR_UNSUPPORTED = -2, /* valid but not implemented: head size, topk above the
                                kernel's limit, pointer not 16-byte aligned */
  TOPK_ERR_CUDA = -3,        /* a CUDA runtime/driver call or a launch failed */
  TOPK_ERR_TIMEOUT = -4,     /* a device pipeline wait ran out its time limit; the
                                kernel stopped early and its outputs are invalid */
  TOPK_ERR_WORKSPACE = -5,   /* an internal consistency check of the selection
                                failed (no input is known to cause it; candidate
                                lists are compacted exactly rather than overflow);
                                outputs invalid */
  TOPK_ERR_NO_DEVICE = -6,   /* no usable sm_103 device */
  TOPK_ERR_SCRATCH_LIMIT = -7 /* the problem needs more scratch than the fixed buffer of
                                 topk_ffn_fwd_noalloc holds */
};

/*
 * Top-k attention forward, Eq. 4 (Sec. 2.2), optionally causal (Eq. 2).
 *   q, k, v, out : device pointers, layouts above, element type `dtype`.
 *   B, H         : batch and heads; every (b, h) is an independent problem.
 *   Lq, Lk       : query and key counts (causal requires Lq <= Lk).
 *   d            : head size.  TOPK_BF16: 64 or 128.  TOPK_F32: 16, 32, 64, 128.
 *   topk         : 1 <= topk <= Lk; the supported maximum is 512.
 *   chunk        : query-chunk size (Sec. 2.2), >= 1; a scheduling hint only.
 *   causal       : 0 or 1.
 *   Scratch: topk_attn_workspace_bytes() (a fixed amount per SM, or none;
 *            plus parts x B*H*Lq x (8 topk + 4) bytes where at most half the
 *            SMs would get a query tile and the key tiles are split into parts).
 * Errors: TOPK_ERR_INVALID_ARG / TOPK_ERR_UNSUPPORTED before any launch;
 *         TOPK_ERR_CUDA if a launch fails (or the scratch cannot be had).
 *         A device-side timeout is not returned by this call (it returns
 *         once the work is enqueued): topk_check() and the *_host calls
 *         report it, from the device's error word (see topk_check).
 */
int topk_attn_fwd(const void* q, const void* k, const void* v, void* out, int B, int H, int Lq, int Lk,
                  int d, int topk, int chunk, int causal, int dtype, void* stream);

/*
 * Same as topk_attn_fwd, and additionally writes, per query row, the kept
 * key indices and their fp32 scores in selection order (score descending,
 * index ascending).  idx [B, H, Lq, topk] int32, -1 padded; score same shape,
 * fp32, -inf padded.  Either may be NULL.  Used for parity checks.
 */
int topk_attn_fwd_indices(const void* q, const void* k, const void* v, void* out, int B, int H, int Lq,
                          int Lk, int d, int topk, int chunk, int causal, int dtype, int32_t* idx,
                          float* score, void* stream);

/*
 * Top-k attention under the general mask of Eq. 2 (Sec. 2.1): B_ij = -inf
 * removes key j from query i's candidates before the top-k.  Three masks
 * combine (a key must pass all of them):
 *   causal  : 0 or 1, as in topk_attn_fwd (key j valid iff j <= i + Lk - Lq).
 *   kv_len  : NULL, or [B] int32 device pointer: key j is valid for every query
 *             of batch b iff j < kv_len[b] (key padding; values are clamped to
 *             [0, Lk]).
 *   mask    : NULL, or a uint32 device bit array: key j is valid for query i of
 *             (b, h) iff bit (j % 32) of word
 *               b * mask_batch_stride + h * mask_head_stride + i * W + j / 32,
 *             W = ceil(Lk / 32), is 1.  A stride of 0 shares the mask across
 *             batches or heads.  4-byte aligned.
 * A row with fewer than k valid keys keeps all of them; a row with none writes
 * zeros.  Other arguments as topk_attn_fwd_indices (idx/score may be NULL).
 * With a bit mask the scores run on the CUDA cores (fp32 FMA of the exact
 * bf16/fp32 inputs); causal and kv_len alone keep the tensor-core kernel.
 * Errors: as topk_attn_fwd; a negative stride is TOPK_ERR_INVALID_ARG, a
 * misaligned mask or kv_len TOPK_ERR_UNSUPPORTED.
 */
int topk_attn_fwd_masked(const void* q, const void* k, const void* v, void* out, int B, int H, int Lq, int Lk,
                         int d, int topk, int chunk, int causal, const int32_t* kv_len, const uint32_t* mask,
                         long long mask_batch_stride, long long mask_head_stride, int dtype, int32_t* idx,
                         float* score, void* stream);

/*
 * Plain (vanilla) attention, Eq. 1 (Sec. 2.1), under Eq. 2's causal mask and
 * per-batch key counts: the softmax covers every valid key.  It is the path
 * the paper compares top-k attention with (Sec. 3; query chunking, Sec. 2.2,
 * bounds its memory there): here the score tile stays on chip, so no
 * [chunk x Lk] buffer exists and `chunk` is validated but has no effect.
 *   q, k, v, out, B, H, Lq, Lk, causal, kv_len: as topk_attn_fwd_masked.
 *   d      : 64 or 128.  dtype: TOPK_BF16 only (fp32 is TOPK_ERR_UNSUPPORTED).
 *   B * H  : at most 65535.
 *   Scratch: topk_vanilla_attn_workspace_bytes() (V transposed, B*H*d*Lk*2
 *   bytes rounded up), from the library's pool.  A row with no valid key
 *   writes zeros.  Errors as topk_attn_fwd.
 */
int topk_vanilla_attn_fwd(const void* q, const void* k, const void* v, void* out, int B, int H, int Lq, int Lk,
                          int d, int chunk, int causal, const int32_t* kv_len, int dtype, void* stream);
size_t topk_vanilla_attn_workspace_bytes(int B, int H, int Lq, int Lk, int d, int dtype);

/*
 * The dense feed-forward layer, Eq. 3 without top-k (Sec. 2.1): out =
 * ReLU(x W1^T) W2, the comparison path for topk_ffn_fwd (Sec. 3).  d_ff is
 * taken in slices of `chunk` keys (chunking bounds the memory, Sec. 2.2): per
 * slice the hidden activations [N, chunk] are formed in bf16, ReLU'd and
 * multiplied into the fp32 output.  The two products run in cuBLAS (plain
 * GEMMs, bf16 inputs, fp32 accumulation); ReLU in the library's own kernel.
 *   x, W1, W2, out, N, d_model, d_ff: as topk_ffn_fwd (d_model a multiple of 8).
 *   chunk  : keys per slice, >= 1; a multiple of 8 unless it covers all of d_ff.
 *   Scratch: topk_vanilla_ffn_workspace_bytes() = N * min(chunk, d_ff) * 2 bytes.
 */
int topk_vanilla_ffn_fwd(const void* x, const void* W1, const void* W2, void* out, int N, int d_model, int d_ff,
                         int chunk, void* stream);
size_t topk_vanilla_ffn_workspace_bytes(int N, int d_model, int d_ff, int chunk);

/*
 * Top-k feed-forward layer, Eq. 3 with the top-k of Eq. 4 and ReLU as the
 * activation (Sec. 2.1, Sec. 2.2).
 *   x  : [N, d_model] bf16 device pointer (the queries).
 *   W1 : [d_ff, d_model] bf16; row j is key j.
 *   W2 : [d_ff, d_model] bf16; row j is value j.
 *   out: [N, d_model] fp32 device pointer.
 *   d_model: a multiple of 64, at most 4096.  1 <= topk <= d_ff, topk <= 1024.
 *   Scratch: topk_ffn_workspace_bytes(); it grows linearly with N.
 * Top-k is taken over the signed scores; ReLU is applied after selection.
 */
int topk_ffn_fwd(const void* x, const void* W1, const void* W2, void* out, int N, int d_model, int d_ff,
                 int topk, void* stream);

/* topk_ffn_fwd plus the kept indices [N, topk] int32 and scores [N, topk] fp32. */
int topk_ffn_fwd_indices(const void* x, const void* W1, const void* W2, void* out, int N, int d_model,
                         int d_ff, int topk, int32_t* idx, float* score, void* stream);

/*
 * Backward pass of top-k attention (Sec. 2.2, "Improving efficiency through
 * top-k attention"): the forward pass caches, per query row, the kept key
 * indices and their scores (topk_attn_fwd_indices writes exactly that
 * cache), and the backward pass recomputes only the activation over them.
 * With L = sum over rows of dout_i . out_i and the kept set held fixed:
 *   a_t  = softmax over the row's kept scores,  da_t = dout_i . v_{j_t},
 *   ds_t = a_t (da_t - sum_u a_u da_u),
 *   dq_i = sum_t ds_t k_{j_t};  dk_j, dv_j = the sums of ds_t q_i and
 *   a_t dout_i over every (i, t) that kept key j of the same (b, h).
 *   q, k, v : the forward pass's inputs (device, `dtype`, layouts above).
 *   dout    : [B, H, Lq, d] device, `dtype` (the dtype of out).
 *   idx     : [B, H, Lq, topk] int32 device, the cached kept indices; an entry
 *             outside [0, Lk) (the forward pass pads with -1) is an empty slot.
 *   score   : [B, H, Lq, topk] fp32 device, the cached scores s_t = q_i . k_{j_t}.
 *   dq      : [B, H, Lq, d] fp32 device (written).
 *   dk, dv  : [B, H, Lk, d] fp32 device (written; keys no row kept get 0).
 *   d       : TOPK_BF16: 64 or 128.  TOPK_F32: 16, 32, 64 or 128.
 *   topk    : the cache's width, 1 <= topk <= 2048.  B*H*Lq*topk and B*H*Lk
 *             must stay below 2^31.
 *   Any order of the kept entries within a row gives the same result.  dk and
 *   dv add each key's terms in an order that depends on atomic ranks, so
 *   they can differ in the last bits from call to call.
 *   Scratch: topk_attn_bwd_workspace_bytes() (20 bytes per cache entry plus
 *   8 bytes per key), from the library's pool.  Errors as topk_attn_fwd.
 */
int topk_attn_bwd(const void* q, const void* k, const void* v, const void* dout, const int32_t* idx,
                  const float* score, float* dq, float* dk, float* dv, int B, int H, int Lq, int Lk, int d,
                  int topk, int dtype, void* stream);

/*
 * Backward pass of the top-k feed-forward layer (Eq. 3 with ReLU, Sec. 2.1
 * and Sec. 2.2) for the cache of topk_ffn_fwd_indices:
 *   a_t = ReLU(s_t),  ds_t = (dout_i . W2_{j_t}) if s_t > 0 else 0,
 *   dx_i = sum_t ds_t W1_{j_t};  dW1_j, dW2_j = the sums of ds_t x_i and
 *   a_t dout_i over every (i, t) that kept key j.
 *   x, W1, W2 : the forward pass's inputs (bf16 device, layouts above).
 *   dout      : [N, d_model] fp32 device (the dtype of the forward output).
 *   idx, score: [N, topk] int32 / fp32 device, the cache.
 *   dx        : [N, d_model] fp32; dW1, dW2: [d_ff, d_model] fp32 (written).
 *   d_model   : a multiple of 64, at most 2048.  1 <= topk <= d_ff.
 *   Scratch: topk_ffn_bwd_workspace_bytes() (20 bytes per cache entry, 4 more per
 *   cache entry and 256 columns of d_model, 8 per key).  Errors as topk_ffn_fwd.
 */
int topk_ffn_bwd(const void* x, const void* W1, const void* W2, const float* dout, const int32_t* idx,
                 const float* score, float* dx, float* dW1, float* dW2, int N, int d_model, int d_ff, int topk,
                 void* stream);

/* Scratch bytes of the two backward calls for these arguments; 0 if invalid or unsupported. */
size_t topk_attn_bwd_workspace_bytes(int B, int H, int Lq, int Lk, int d, int topk, int dtype);
size_t topk_ffn_bwd_workspace_bytes(int N, int d_model, int d_ff, int topk);

/*
 * topk_ffn_fwd without any device allocation.  The paper has no counterpart:
 * this entry exists for callers that cannot allocate device memory when they
 * call -- for instance a host runtime that hands out all device memory from
 * its own arena and allows no other allocation, or a latency-bound serving
 * loop that must never wait on an allocator or fail on a fragmented pool.
 * Instead of taking scratch from the stream-ordered pool it uses one buffer
 * of TOPK_FFN_NOALLOC_SCRATCH_BYTES that is part of the library: every GPU
 * that loads libtopk.so holds it until the process exits.
 *   - Arguments, layouts and results are those of topk_ffn_fwd; the caller
 *     still passes (and owns) x, W1, W2 and out.
 *   - Returns TOPK_ERR_SCRATCH_LIMIT, before launching anything, when
 *     topk_ffn_workspace_bytes() of the arguments exceeds the buffer.
 *   - The first call on a device looks up the buffer's device address (one
 *     runtime query, no allocation); make that first call before any stream
 *     capture on that device.
 *   - All calls on a device share the one buffer, and each call re-clears
 *     the parts that must start at zero.  Calls whose work overlaps on the
 *     GPU (other streams, or other threads) race on the buffer: serialise
 *     them, e.g. by issuing them on one stream.
 * It calls no cudaMalloc, cudaFree or other allocating routine.
 */
#define TOPK_FFN_NOALLOC_SCRATCH_BYTES (32u << 20)
int topk_ffn_fwd_noalloc(const void* x, const void* W1, const void* W2, void* out, int N, int d_model,
                         int d_ff, int topk, void* stream);

/* Bytes of stream-ordered scratch the calls above take for these arguments
 * (0 if none).  Returns 0 as well when the arguments are invalid.
 *   - attention: the bf16 tensor-core kernel with split selection parks each
 *     work unit's kept keys for its epilogue warps: per CTA (one per SM, at
 *     most one per 128-query tile) 4 x 2 x topk x 32 keys of 8 bytes plus
 *     256 counts of 4 bytes, whatever Lq and Lk are.  Sized for the current
 *     device, or for 152 SMs (a GB300) when no device is visible.
 *   - feed-forward: linear in N (see topk_ffn_fwd). */
size_t topk_attn_workspace_bytes(int B, int H, int Lq, int Lk, int d, int topk, int chunk, int dtype);
size_t topk_ffn_workspace_bytes(int N, int d_model, int d_ff, int topk);

/*
 * End-to-end variants taking HOST pointers (pinned memory is fastest).  They
 * stage the inputs into device memory from the library's pool, run the call
 * above on `stream`, copy the result back and synchronise `stream` before
 * returning.  Sizes and dtypes as above.
 *   - topk_attn_fwd_host splits the B*H heads into up to 8 consecutive
 *     slices when there are enough query tiles (about 6 per SM per slice)
 *     and launches one call per slice, alternating between two compute
 *     streams of the library (ordered after `stream`); each slice's inputs
 *     are copied on a copy stream of the library and its output copied back
 *     on another.  The copies of neighbouring slices overlap the kernels,
 *     and a slice's kernel starts on the SMs the previous slice's last wave
 *     leaves idle.  The result is identical to one call over all heads.
 *   - topk_ffn_fwd_host copies x and W1 first and W2 on a copy stream while
 *     the score and selection kernels run; the W2 gather waits for it.
 *   The library's streams are shared by all host-buffer calls on a device;
 *   `stream` is synchronised, after it has waited for all of them.
 */
int topk_attn_fwd_host(const void* q, const void* k, const void* v, void* out, int B, int H, int Lq,
                       int Lk, int d, int topk, int chunk, int causal, int dtype, void* stream);
int topk_ffn_fwd_host(const void* x, const void* W1, const void* W2, void* out, int N, int d_model,
                      int d_ff, int topk, void* stream);

/* Synchronises `stream` and returns the device-side error recorded since the
 * last check (TOPK_ERR_TIMEOUT before TOPK_ERR_WORKSPACE), clearing it;
 * TOPK_ERR_CUDA if the stream itself reports an error; else TOPK_OK.
 * The error word is ONE per device, shared by every stream and host thread
 * that calls into the library on that device: an error raised by work on one
 * stream is reported to (and cleared by) whichever caller checks first, and
 * the *_host calls check it too.  Callers that share a device and need to
 * tell their errors apart must serialise their calls and checks. */
int topk_check(void* stream);

/* Human-readable text for a return code (static storage). */
const char* topk_error_string(int code);

/* Number of kernel launches the last successful call on this host thread
 * enqueued (for launch accounting in benchmarks). */
int topk_last_launch_count(void);

/* Testing hook: sets the device-side wait limit in microseconds for later
 * calls (0 restores the default of 2 s) and returns the previous value. */
long long topk_set_wait_limit_us(long long us);

/* Device memory of the library's own stream-ordered pool on the current
 * device (scratch of the device-pointer calls, staging buffers of the *_host
 * calls): *used_high = the most bytes in use at once since the last reset,
 * *reserved = bytes the pool holds now (in use or kept for later calls).
 * Either pointer may be NULL; reset_high != 0 restarts the high-water mark
 * after reading it.  Returns TOPK_ERR_NO_DEVICE without a usable device. */
int topk_pool_usage(size_t* used_high, size_t* reserved, int reset_high);

/* Hands the pool's reserved but unused memory back to the device.  Memory
 * freed by enqueued work is released only once that work has completed:
 * synchronise the streams that used the library first. */
int topk_pool_trim(void);

/* Testing hook: when `on` is non-zero, later tcgen05 attention launches
 * withhold their second key tile, so that the consumers' bounded waits run
 * out and the call reports TOPK_ERR_TIMEOUT through topk_check() without
 * hanging the device.  Returns the previous setting. */
int topk_debug_skip_arrive(int on);

#ifdef __cplusplus
}
#endif

#endif /* TOPK_ATTENTION_H */
