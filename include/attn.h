/*
 * attn.h -- C ABI of the GB300 (sm_103a) three-stage attention library.
 *
 * The library implements the per-layer attention block of the paper's three
 * static-shape stages (arxiv 2607.15865, Section 4; Table 1):
 *
 *   prefill     a prompt of chunk_len tokens attends causally to itself
 *               (Section 4.2, with_history=False; Listing 1);
 *   prefill_kv  a chunk of chunk_len new tokens attends to hist_len history
 *               tokens already in the cache plus itself, causally
 *               (Section 4.3, with_history=True; Listing 2);
 *   decode      one new token per sequence attends to the hist_len[b] valid
 *               tokens of a static-maximum-length cache plus itself
 *               (Section 4.4; the runtime-filled mask is given as lengths).
 *
 * Every stage rotates q and k with RoPE using cos/sin gathered from a table
 * precomputed per position (Listing 1 "Gather"/"Rope"; Section 4.6.2), writes the
 * rotated k and the unchanged v of the new tokens into the caller's cache in
 * place (Listing 2 "Concat"; Section 4.6.3), and computes scaled dot-product
 * attention with scale 1/sqrt(head_dim) (FAttention, Section 2.2) under the
 * causal mask (Section 4.6.1).  Grouped-query attention: query head h reads kv
 * head h / (n_q_heads / n_kv_heads).
 *
 * Numerics: the table holds cos/sin of p*theta^(-2j/D) (element j paired with
 * j + D/2) computed in double and rounded to float; RoPE runs in float and the
 * rotated q and k are rounded to bf16 (nearest even); scores, softmax and the
 * value sum accumulate in float; out is rounded to bf16 (nearest even).
 *
 * Data types and layouts.  "bf16" below is a pointer to bf16 values given as
 * their 16-bit patterns (uint16_t), all in device memory, densely packed:
 *   q    [batch, chunk_len, n_q_heads,  head_dim]
 *   k, v [batch, chunk_len, n_kv_heads, head_dim]
 *   k_cache, v_cache [batch, n_kv_heads, max_len, head_dim]
 *   out  [batch, chunk_len, n_q_heads,  head_dim]
 * Decode uses chunk_len = 1.  All device pointers must be 16-byte aligned.
 *
 * Ownership.  The caller owns every device buffer passed to a call.  The
 * context owns only its own device memory: the RoPE tables (2 x max_len x
 * head_dim/2 floats, held twice: position-major and in groups of four pairs), the decode
 * split-KV partials (batch x n_q_heads x 256 x (head_dim + 2) floats) and counters
 * (5 x batch x n_kv_heads x 16 + 1 ints: one set per column group of the multi-token
 * decode), the prefill partials of split work (SM count x 256 x (head_dim + 2)
 * floats), the q, k, v and attention output of one decode block (attn_decode_layer)
 * and a device error word; all allocated by attn_create
 * and freed by attn_destroy.  No stage call allocates, frees or synchronises: each one only
 * enqueues kernels on `stream` and returns.  Calls that use the same context
 * share its scratch buffers, so they must not run concurrently on different
 * streams.
 *
 * Errors.  Every int-returning call returns ATTN_OK (0) or a negative code and
 * writes nothing when it rejects its arguments; that includes shapes whose launch
 * would exceed a grid limit (a decode with batch x column groups, or head_dim 64
 * kv heads x head passes, above 65535; a prefill chunk whose pairs of 128-row
 * query tiles x n_q_heads x batch exceed 2^30).  Launch failures return
 * ATTN_ECUDA (attn_last_cuda_error_string() gives the runtime's text).  The
 * decode lengths live on the device, so a decode whose hist_len[b] is outside
 * [0, max_len - 1] cannot be rejected on the host: the kernels then skip
 * sequence b (its cache and out are not written) and set a bit in the context's
 * device error word, which attn_device_error() reads.  No kernel traps.
 */
#ifndef ATTN_GB300_ATTN_H
#define ATTN_GB300_ATTN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ATTN_OK 0
#define ATTN_EINVAL (-1)   /* invalid argument or unsupported shape */
#define ATTN_EARCH (-2)    /* current device is not compute capability 10.3 (sm_103) */
#define ATTN_ECUDA (-3)    /* a CUDA runtime or launch error */
#define ATTN_ENOMEM (-4)   /* device memory allocation failed in attn_create */
#define ATTN_EDEVICE (-5)  /* attn_device_error found the device error word set */

/* Bits of the device error word. */
#define ATTN_DEVERR_HIST_RANGE 1 /* a decode hist_len[b] was outside [0, max_len - 1] */
#define ATTN_DEVERR_TIMEOUT 2    /* a pipeline wait inside a kernel exceeded its time limit (about 1 s);
                                    the affected outputs are not written */

/* Opaque CUDA stream handle; pass a cudaStream_t (0 = legacy default stream). */
typedef struct CUstream_st* attn_stream_t;

typedef struct attn_cfg {
    int batch;       /* sequences per call, >= 1 */
    int n_q_heads;   /* query heads Hq, a multiple of n_kv_heads */
    int n_kv_heads;  /* key/value heads Hkv; group size Hq/Hkv must be <= 16 */
    int head_dim;    /* D: 64 or 128 */
    int max_len;     /* static maximum cache length L (positions 0 .. L-1), 1 .. 1<<20 */
    double rope_theta; /* RoPE base theta > 0 */
} attn_cfg;

typedef struct attn_ctx attn_ctx;

/*
 * Create a context for one shape on the current CUDA device.  Validates cfg,
 * checks that the device is sm_103, builds the RoPE tables (Section 4.6.2) and
 * allocates the context's scratch.  *out receives the context on success and
 * NULL otherwise.  Returns ATTN_OK, ATTN_EINVAL, ATTN_EARCH, ATTN_ENOMEM or
 * ATTN_ECUDA.  Blocking (it uploads the tables).
 */
int attn_create(const attn_cfg* cfg, attn_ctx** out);

/* Free a context and its device memory (blocking).  NULL is ignored. */
void attn_destroy(attn_ctx* ctx);

/*
 * Prefill (Section 4.2): positions 0 .. chunk_len-1.  Writes cache slots
 * [0, chunk_len) of every sequence and out.  1 <= chunk_len <= max_len.
 */
int attn_prefill(attn_ctx* ctx, const uint16_t* q, const uint16_t* k, const uint16_t* v, int chunk_len,
                 uint16_t* k_cache, uint16_t* v_cache, uint16_t* out, attn_stream_t stream);

/*
 * Prefill_kv (Section 4.3): the caches hold hist_len valid history tokens in
 * slots [0, hist_len) of every sequence; the new tokens take positions
 * hist_len .. hist_len+chunk_len-1 and slots of the same index.  Only those
 * slots are written.  hist_len >= 0, chunk_len >= 1, hist_len + chunk_len <= max_len.
 * With hist_len = 0 the result equals attn_prefill (Section 4.2: one template).
 */
int attn_prefill_kv(attn_ctx* ctx, const uint16_t* q, const uint16_t* k, const uint16_t* v, int hist_len,
                    int chunk_len, uint16_t* k_cache, uint16_t* v_cache, uint16_t* out,
                    attn_stream_t stream);

/*
 * Decode (Section 4.4): one new token per sequence.  d_hist_len is a device
 * array [batch] of int32: sequence b has hist_len[b] valid tokens in slots
 * [0, hist_len[b]); its new token is written to slot hist_len[b] and attends to
 * slots [0, hist_len[b]].  q [batch,1,Hq,D], k/v [batch,1,Hkv,D], out [batch,1,Hq,D].
 * Out-of-range lengths: see "Errors" above.
 */
int attn_decode(attn_ctx* ctx, const uint16_t* q, const uint16_t* k, const uint16_t* v,
                const int32_t* d_hist_len, uint16_t* k_cache, uint16_t* v_cache, uint16_t* out,
                attn_stream_t stream);

/*
 * Multi-token decode: n_new tokens per sequence in one call (Section 4.4 with more than
 * one new token, e.g. to verify a speculative draft; the paper names speculative
 * decoding as future work, Section 6).  Sequence b's token i takes position
 * hist_len[b] + i, is written to that slot and attends to slots [0, hist_len[b] + i]
 * (causal among the new tokens); lengths are per sequence, read on the device.
 *   q [batch, n_new, Hq, D], k/v [batch, n_new, Hkv, D], out [batch, n_new, Hq, D].
 * head_dim 128: 1 <= n_new <= 16 (ATTN_EINVAL otherwise).  The n_new * (Hq / Hkv)
 * (query head, token) columns of a kv head run in groups of 16, one group per CTA of a key
 * range; the groups of one range read the same cache tiles at about the same time, so the
 * repeats come from L2 while the history fits there.  A sequence whose hist_len[b] + n_new
 * exceeds max_len is skipped and flagged as in attn_decode.
 * head_dim 64: 1 <= n_new <= max_len; the tokens run as n_new attn_decode steps in order
 * (token t at hist_len[b] + t, the same result), each step's rows copied in and out of the
 * context's buffers, so the history is streamed n_new times; a token whose position passes
 * max_len - 1 is flagged and skipped as one attn_decode step would (the tokens before it in
 * that sequence are computed).  n_new = 1 is attn_decode.
 */
int attn_decode_multi(attn_ctx* ctx, const uint16_t* q, const uint16_t* k, const uint16_t* v,
                      const int32_t* d_hist_len, int n_new, uint16_t* k_cache, uint16_t* v_cache, uint16_t* out,
                      attn_stream_t stream);

/*
 * Stage driver, long prompts (Section 4.1, the third scenario: a prompt longer than
 * the stages' static chunk length runs as 1 prefill + N prefill_kv).  The prompt's
 * prompt_len tokens take positions hist_len .. hist_len+prompt_len-1.  They are
 * processed in segments of seg_len tokens (the last one may be shorter), in order:
 * the first segment by attn_prefill when hist_len = 0 and by attn_prefill_kv
 * otherwise (a later session of a conversation, Section 4.1 scenario 2), every
 * further segment by attn_prefill_kv over all positions before it.
 *   q   [batch, prompt_len, n_q_heads,  head_dim]   (the whole prompt, dense)
 *   k,v [batch, prompt_len, n_kv_heads, head_dim]
 *   out [batch, prompt_len, n_q_heads,  head_dim]
 * Cache slots [hist_len, hist_len+prompt_len) are written.  The result equals
 * one attn_prefill_kv of the whole prompt up to the order of float accumulation.
 * hist_len >= 0, prompt_len >= 1, seg_len >= 1, hist_len + prompt_len <= max_len;
 * otherwise ATTN_EINVAL before any launch.  A launch failure in segment i returns
 * ATTN_ECUDA with the earlier segments enqueued.
 */
int attn_prompt(attn_ctx* ctx, const uint16_t* q, const uint16_t* k, const uint16_t* v, int hist_len,
                int prompt_len, int seg_len, uint16_t* k_cache, uint16_t* v_cache, uint16_t* out,
                attn_stream_t stream);

/*
 * Stage driver, decode loop (Section 4.5, steps 3-5, the attention part): n_steps
 * decode steps in a row.  Step t's token of sequence b takes position
 * d_hist_len[b] + t and attends to slots [0, d_hist_len[b] + t]; d_hist_len is
 * read, not written.  Inputs are step-major so that each step's operands are
 * those of one attn_decode:
 *   q   [n_steps, batch, 1, n_q_heads,  head_dim]
 *   k,v [n_steps, batch, 1, n_kv_heads, head_dim]
 *   out [n_steps, batch, 1, n_q_heads,  head_dim]
 * 1 <= n_steps <= max_len.  A position past max_len - 1 is handled as in
 * attn_decode (that step skips the sequence and sets ATTN_DEVERR_HIST_RANGE).  Like
 * every stage call it only enqueues kernels, so a serving loop can capture it into
 * a CUDA graph once and replay it.
 */
int attn_decode_steps(attn_ctx* ctx, const uint16_t* q, const uint16_t* k, const uint16_t* v,
                      const int32_t* d_hist_len, int n_steps, uint16_t* k_cache, uint16_t* v_cache,
                      uint16_t* out, attn_stream_t stream);

/*
 * Synchronise `stream`, read and clear the context's device error word.
 * *flags (may be NULL) receives the ATTN_DEVERR_* bits.  Returns ATTN_OK when
 * the word was zero, ATTN_EDEVICE when a bit was set, ATTN_ECUDA on a CUDA error.
 */
int attn_device_error(attn_ctx* ctx, attn_stream_t stream, int* flags);

/*
 * Failure detection (no counterpart in the paper, which runs on a static TPU schedule):
 * every wait inside a kernel of this library -- on a copy, a tensor-core result or a
 * hand-over between the kernel's warps -- gives up after a time limit, records
 * ATTN_DEVERR_TIMEOUT in the device error word, lets the copies and MMAs it has already
 * issued finish, releases its tensor memory and returns; nothing spins forever and
 * nothing traps, so the context stays usable.
 *
 * attn_set_wait_limit sets that limit for the kernels this context launches from the
 * next call on: limit_ns > 0 is the limit in nanoseconds, limit_ns <= 0 restores the
 * default of 1 s.  The waits that drain copies and MMAs already in flight always keep
 * the default.  With a limit far below a kernel's latency (a test of the failure path)
 * the next stage calls give up at their first wait that is not already satisfied: the
 * error word gets ATTN_DEVERR_TIMEOUT, and their outputs and the cache slots they would
 * have written are undefined (every other cache slot is left as it was).  Restore the
 * default and read the error word (attn_device_error) before relying on results again.
 * Returns ATTN_OK, or ATTN_EINVAL for a null context.  Host-only; enqueues nothing.
 */
int attn_set_wait_limit(attn_ctx* ctx, long long limit_ns);

/*
 * Kernel timing (tracing).  The attention entry points launch these kernels (the
 * W4BF16 kernels, which take no context, are not timed):
 *   ATTN_KERNEL_ROPE_APPEND     RoPE of the new keys + in-place cache append (every stage)
 *   ATTN_KERNEL_FLASH_FWD       causal flash attention (prefill, prefill_kv), with the
 *                               merge kernel of its split tail when it runs one
 *   ATTN_KERNEL_DECODE_SPLIT    split-KV decode (decode); with head_dim 128 it also
 *                               merges the splits and writes out itself
 *   ATTN_KERNEL_DECODE_COMBINE  log-sum-exp merge of the partials (decode, head_dim 64)
 * (ATTN_KERNEL_FLASH_FWD also covers the small merge kernel that follows it when
 * the last round of its work is split across CTAs; both count as launches.)
 * attn_timing_enable(ctx, n) creates n pairs of CUDA events (blocking, the only
 * allocation it makes) and from then on every stage call records one pair
 * around each kernel it enqueues, on the call's stream; n = 0 disables timing
 * and frees the events.  Launches beyond n pairs are counted but not timed.
 * attn_timing_read synchronises the device, adds up the elapsed time of every
 * recorded pair per kernel into ms[ATTN_NUM_KERNELS] and the launches counted
 * since the last read (timed or not, enabled or not) into
 * launches[ATTN_NUM_KERNELS], then starts a new period.  Either array may be
 * NULL.  Both return ATTN_OK, ATTN_EINVAL or ATTN_ECUDA.
 */
#define ATTN_KERNEL_ROPE_APPEND 0
#define ATTN_KERNEL_FLASH_FWD 1
#define ATTN_KERNEL_DECODE_SPLIT 2
#define ATTN_KERNEL_DECODE_COMBINE 3
#define ATTN_NUM_KERNELS 4
int attn_timing_enable(attn_ctx* ctx, int max_launches);
int attn_timing_read(attn_ctx* ctx, double* ms, long long* launches);

/*
 * Decode for callers that cannot allocate device memory.  The paper has no
 * counterpart to this entry point; it exists for the library's users.
 *
 * Some callers cannot call cudaMalloc: code running inside a framework that owns
 * all device memory and hands out only its own pre-reserved buffers, processes
 * whose device memory is provisioned once up front, or callbacks that must not
 * enter the allocator.  They cannot use attn_create, which allocates.  This call
 * computes exactly what attn_decode computes, with no context and no allocation:
 *   - the caller passes every input and output, including the RoPE tables d_cos,
 *     d_sin (float [max_len][head_dim/2], row p column j holding cos / sin of
 *     p * theta^(-2j/head_dim) evaluated in double and rounded to float -- the
 *     table attn_create builds) and d_err, an int32 the caller zeroes and reads
 *     back (it receives the ATTN_DEVERR_* bits, as attn_device_error reports);
 *   - the split-KV partials live in a static device array of
 *     ATTN_NOALLOC_SCRATCH_FLOATS floats (4 MiB) that every GPU which loads this
 *     library holds until the process exits, beside 40961 int counters
 *     (160 KiB).  Shapes whose partials do not fit even with one split
 *     (batch * n_q_heads * (head_dim + 2) > that size) are rejected with
 *     ATTN_EINVAL; larger ones use fewer splits.
 * All calls share those arrays.  Nothing in the partials has to start at zero
 * (every call rewrites the part it reads); the counters are zero when the
 * library loads and every completed call leaves them zero.  Calls whose kernels
 * overlap on the GPU --
 * on different streams, or from several threads -- race on it and must be
 * serialised by the caller.  The first call on each device looks up the array's
 * device address (cudaGetSymbolAddress, with that device current) and caches
 * it; make that first call before any stream capture.  cudaDeviceReset discards
 * that set-up (the array and the kernels' attributes are reloaded with new
 * addresses), so a process that resets a device must not call this entry point on
 * it afterwards.  A call whose kernels were abandoned part-way (a stream torn down
 * while they ran) leaves the shared counters undefined until the process exits;
 * a wait that ran out (ATTN_DEVERR_TIMEOUT) does not: those kernels still finish
 * and clear them.  The other arguments and the errors are those of attn_decode
 * (an ATTN_ECUDA leaves its text for attn_last_cuda_error_string); cfg is read on
 * the host only.
 */
#define ATTN_NOALLOC_SCRATCH_FLOATS (1 << 20)
int attn_decode_noalloc(const attn_cfg* cfg, const float* d_cos, const float* d_sin, const uint16_t* q,
                        const uint16_t* k, const uint16_t* v, const int32_t* d_hist_len, uint16_t* k_cache,
                        uint16_t* v_cache, uint16_t* out, int32_t* d_err, attn_stream_t stream);

/* W4BF16 weight-only matrix-vector product of the decode stage (Section 5.1: the
 * models run with 4-bit weights and bf16 activations; Section 5.2: decode speed is
 * the rate at which the weights stream from memory).  For m < M, n < N:
 *   y[m][n] = bf16( sum_{k<K} x[m][k] * (q[n][k] - z[n][k/128]) * s[n][k/128] )
 * with the sum formed in float (products exact, sums rounded), y rounded to nearest.
 *   w_tiles device, 16-byte aligned: the [N, K] weight matrix as ceil(N/16) * (K/128)
 *           records of ATTN_W4_TILE_BYTES (1072) bytes, record T * (K/128) + G holding
 *           rows 16T..16T+15 of input group G (k = 128G .. 128G+127):
 *             bytes    0..1023  codes, tile row r at byte 64 r as 16 little-endian uint32
 *                               words; word i holds k = 128G + 8i + j (j = 0..7), the
 *                               4-bit code of j at bit (0,16,4,20,8,24,12,28)[j];
 *             bytes 1024..1055  the 16 rows' scales s, bf16, row r at byte 1024 + 2r;
 *             bytes 1056..1071  the 16 rows' zero points z (0..15), row r at 1056 + r.
 *           Rows past N in the last row-tile are ignored.
 *   x       device, bf16 [M][K], 16-byte aligned.   y: device, bf16 [M][N].
 *   d_err   device int32 or NULL: a wait of the kernel that runs out (a copy that never
 *           lands) sets ATTN_DEVERR_TIMEOUT in it and leaves y undefined.
 *   flags   0 or ATTN_W4_WEIGHTS_STATIC.  The kernel is launched as a programmatic
 *           dependent of the kernel before it on `stream`: it reads x and writes y only
 *           after that kernel has finished, and lets the kernel after it begin early.
 *           With ATTN_W4_WEIGHTS_STATIC it also starts reading w_tiles before the
 *           previous kernel has finished, so a chain of calls streams the next matrix
 *           during the previous call's last CTAs: set it only when the kernel right
 *           before this call on the stream does not write w_tiles.
 * K a positive multiple of 128 with attn_w4bf16_rows_per_launch(K) >= 1; any M >= 1,
 * N >= 1.  One launch serves attn_w4bf16_rows_per_launch(K) rows of x (x is staged in
 * shared memory); further rows take further passes over the weights.  Enqueued on
 * `stream`; nothing is allocated or synchronised; buffers stay the caller's.
 * Returns ATTN_OK, ATTN_EINVAL (null pointer, bad size, alignment or flag), ATTN_EARCH
 * or ATTN_ECUDA. */
#define ATTN_W4_TILE_BYTES 1072
#define ATTN_W4_WEIGHTS_STATIC 1
int attn_w4bf16_gemv(const void* w_tiles, const uint16_t* x, int M, int N, int K, uint16_t* y, int32_t* d_err,
                     int flags, attn_stream_t stream);

/* attn_w4bf16_gemv with the parts of Listing 1's block around the product fused in (each
 * optional):
 *   rms_gamma  NULL, or device bf16 [K], 8-byte aligned: x is replaced by RMSNorm(x):
 *              x * r * gamma rounded to bf16, r = 1 / sqrt(mean over k of x^2 + rms_eps),
 *              in float, per row of x (0 <= rms_eps < 1);
 *   residual   NULL, or device bf16 [M][N]: added to the product in float before the
 *              rounding of y (when y is not split it may be y itself: each element is read
 *              before it is written);
 *   y1, y2     NULL (y is [M][N]), or both set with 0 < n_split0 < n_split1 < N: columns
 *              [0, n_split0) go to y as [M][n_split0], [n_split0, n_split1) to y1 as
 *              [M][n_split1 - n_split0] and [n_split1, N) to y2 as [M][N - n_split1] (q, k
 *              and v of a stacked QKV projection).
 * The other arguments and the errors are those of attn_w4bf16_gemv. */
int attn_w4bf16_gemv_fused(const void* w_tiles, const uint16_t* x, int M, int N, int K, const uint16_t* rms_gamma,
                           float rms_eps, const uint16_t* residual, uint16_t* y, int n_split0, uint16_t* y1,
                           int n_split1, uint16_t* y2, int32_t* d_err, int flags, attn_stream_t stream);

/* One decode step of the attention half of a decoder block (Listing 1: input_layernorm,
 * q/k/v projections, RoPE, attention, o_proj + residual) with W4BF16 weights, for the
 * context's shape (B = batch sequences, one new token each):
 *   x           device bf16 [B][hidden], 16-byte aligned: the block's input (residual stream);
 *   rms_gamma   device bf16 [hidden], 8-byte aligned; rms_eps: see attn_w4bf16_gemv_fused;
 *   wqkv_tiles  the tile stream (attn_w4bf16_gemv) of the stacked [(Hq + 2 Hkv) D, hidden]
 *               matrix: rows of q_proj, then k_proj, then v_proj;
 *   wo_tiles    the tile stream of o_proj, [hidden, Hq D];
 *   hidden      a multiple of 128 (as is Hq D);
 *   d_hist_len, k_cache, v_cache: as in attn_decode (the new k and v are appended);
 *   h_out       device bf16 [B][hidden]: x + o_proj(attention); may be x itself.
 * q, k, v and the attention output live in buffers of the context; the step enqueues the
 * fused QKV GEMV, the decode kernels and the o_proj GEMV on `stream` (flags applies to the
 * QKV GEMV, as in attn_w4bf16_gemv; the o_proj GEMV always streams its weights early).  A
 * GEMV wait that runs out sets ATTN_DEVERR_TIMEOUT in the context's error word
 * (attn_device_error).  Returns ATTN_OK, ATTN_EINVAL, ATTN_EARCH or ATTN_ECUDA. */
int attn_decode_layer(attn_ctx* ctx, const uint16_t* x, const uint16_t* rms_gamma, float rms_eps,
                      const void* wqkv_tiles, const void* wo_tiles, int hidden, const int32_t* d_hist_len,
                      uint16_t* k_cache, uint16_t* v_cache, uint16_t* h_out, int flags, attn_stream_t stream);

/*
 * The attention half of a decoder block for a prefill (hist_len = 0, Section 4.2) or
 * prefill_kv (Section 4.3) chunk, with W4BF16 weights (Listing 1's dataflow):
 *   xn = bf16(x * r * rms_gamma), r = 1 / sqrt(mean(x^2) + rms_eps)    per token
 *   q | k | v = bf16(xn . Wqkv^T)        each weight rounded once to bf16 (attn_w4bf16_gemm)
 *   out = the prefill_kv stage of q, k, v over hist_len history tokens (RoPE, in-place
 *         cache append at slots hist_len .. hist_len + chunk_len - 1, causal GQA attention)
 *   h_out = bf16(x + out . Wo^T)
 *   x, h_out   device bf16 [batch][chunk_len][hidden], 16-byte aligned; h_out may be x
 *   rms_gamma  device bf16 [hidden];  rms_eps >= 0, finite
 *   wqkv_tiles the tile stream (attn_w4bf16_gemv's format) of the stacked
 *              [(n_q_heads + 2 n_kv_heads) head_dim, hidden] matrix: q_proj rows, then
 *              k_proj, then v_proj;  wo_tiles: that of the [hidden, n_q_heads head_dim] o_proj
 *   k_cache, v_cache as for attn_prefill_kv
 *   workspace  device memory of at least attn_prefill_layer_workspace(ctx, hidden,
 *              chunk_len) bytes, 256-byte aligned, owned by the caller (the normalised x,
 *              q, k, v and the attention output live there; nothing is allocated)
 * hidden, n_q_heads head_dim and (n_q_heads + 2 n_kv_heads) head_dim multiples of 128;
 * 1 <= chunk_len, hist_len + chunk_len <= max_len, batch * chunk_len <= 65535 * 128.
 * Enqueues four launches on `stream` (RMSNorm, QKV GEMM, attention, o_proj GEMM); a
 * wait that runs out sets ATTN_DEVERR_TIMEOUT in the context's error word.  Returns
 * ATTN_OK, ATTN_EINVAL, ATTN_EARCH or ATTN_ECUDA.
 */
size_t attn_prefill_layer_workspace(const attn_ctx* ctx, int hidden, int chunk_len);
int attn_prefill_layer(attn_ctx* ctx, const uint16_t* x, const uint16_t* rms_gamma, float rms_eps,
                       const void* wqkv_tiles, const void* wo_tiles, int hidden, int hist_len, int chunk_len,
                       uint16_t* k_cache, uint16_t* v_cache, uint16_t* h_out, void* workspace,
                       size_t workspace_bytes, attn_stream_t stream);

/* W4BF16 weight GEMM of the prefill-side projections (Listing 1's q/k/v/o_proj over a
 * chunk of T tokens; Section 5.1 W4BF16), on the tensor cores:
 *   y[t][n] = bf16( sum_{k<K} x[t][k] * W[n][k] ),  W[n][k] = bf16((q - z) * s)
 * each weight rounded once to bf16 (the decode-then-multiply reading), f32 sums.
 *   w_tiles  the tile stream of the [N, K] matrix (format of attn_w4bf16_gemv);
 *   x        device bf16 [T][K], 16-byte aligned;  y: device bf16 [T][N], 16-byte aligned;
 *   d_err    device int32 or NULL: a wait that runs out sets ATTN_DEVERR_TIMEOUT in it.
 * 1 <= T <= 65535 * 128; N and K positive multiples of 128.  Enqueued on `stream`;
 * nothing is allocated or synchronised.  Returns ATTN_OK, ATTN_EINVAL, ATTN_EARCH or
 * ATTN_ECUDA. */
int attn_w4bf16_gemm(const void* w_tiles, const uint16_t* x, int T, int N, int K, uint16_t* y, int32_t* d_err,
                     attn_stream_t stream);

/* Rows of x one attn_w4bf16_gemv launch serves for inner size K: 8, 4, 2 or 1, or 0
 * when K is not a positive multiple of 128 or too large to stage (host only). */
int attn_w4bf16_rows_per_launch(int K);

/* Static text for an ATTN_* code. */
const char* attn_strerror(int code);

/* Text of the most recent CUDA error seen by this library on the calling thread. */
const char* attn_last_cuda_error_string(void);

#ifdef __cplusplus
}
#endif

#endif /* ATTN_GB300_ATTN_H */
