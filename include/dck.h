/*
 * dck.h - C ABI of libdck: decode attention over a DynaCalKV compressed KV cache
 * on NVIDIA GB300 (sm_103a).
 *
 * The method (DynaCalKV, arXiv 2607.24331):
 *   Sec. III-A  a rank-r factorisation W ~ L R caches z = x L (r numbers per
 *               token) instead of x W and rebuilds x W ~ z R at attention time.
 *   Sec. III-C  the key projection is split column-wise into head groups of
 *               varying size; group g keeps its own factors L_g (D x r_g) and
 *               R_g (r_g x n_g*d), so each token caches one key latent
 *               c_t^g = x_t L_g per group, of rank r_g.
 *   Sec. III-D  the value projection is factorised as a whole, W^(v) ~ L_v R_v,
 *               so each token caches one value latent v_t = x_t L_v of rank r_v.
 * Here A_g = L_g, B_g = R_g, A_v = L_v and B_v = R_v.
 *
 * Decode attention (one query per sequence, at position L_b - 1, the decode
 * step's own token being the last cache row): for query head j with KV head
 * h = floor(j * Hkv / Hq) in group g at column-block slot s,
 *   k_t   = c_t^g B_g[:, s*d:(s+1)*d],  RoPE (rotate-half pairs (i, i+d/2),
 *           omega_i = theta^(-2i/d)) at position t; q_j rotated at L_b - 1;
 *   p     = softmax_t(<q_j', k_t'> / sqrt(d));
 *   o_j   = (sum_t p_t v_t) B_v[:, h*d:(h+1)*d]
 * (values are absorbed in latent space: sum_t p_t (v_t B_v) = (sum_t p_t v_t) B_v).
 * The paper describes neither decode nor RoPE; these conventions are the
 * library's and are stated here in full.
 *
 * Conventions of every entry point
 *   - Pointers named d_* and all tensor pointers are DEVICE pointers on the
 *     current CUDA device; descriptor arrays are HOST pointers, read during
 *     the call only.
 *   - The caller owns every buffer, including the workspace.  No entry point
 *     allocates device memory or synchronises the stream; all work is
 *     enqueued on `stream` (a cudaStream_t; NULL = legacy default stream).
 *   - Host-side validation failures return a negative status before any
 *     launch.  A failed launch returns DCK_ERR_CUDA.  Device-side checks
 *     (lengths and rows outside the cache) record an error word that
 *     dck_last_device_error() reports; the offending sequence is treated as
 *     empty and its output is zero.
 *   - No exception crosses the ABI.  Calls on distinct streams may run
 *     concurrently if they use distinct workspaces.
 *   - Tensors are dense row-major; element type is the descriptor's dtype
 *     (bf16 or fp32) unless stated otherwise.
 */
#ifndef DCK_H_
#define DCK_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  DCK_OK = 0,
  DCK_ERR_INVALID = -1,     /* null pointer, bad size, malformed descriptor */
  DCK_ERR_UNSUPPORTED = -2, /* well-formed but outside what the kernels implement */
  DCK_ERR_WORKSPACE = -3,   /* workspace missing or smaller than the size query */
  DCK_ERR_CUDA = -4,        /* a CUDA runtime call or kernel launch failed */
  DCK_ERR_TIMEOUT = -5      /* a bounded device-side wait gave up */
} dck_status;

typedef enum { DCK_BF16 = 0, DCK_F32 = 1 } dck_dtype;

/*
 * One attention layer with a DynaCalKV cache (Sec. III-C key groups,
 * Sec. III-D whole-matrix value factor).
 *   hidden        D, the model width (rows of A_k and A_v)
 *   n_q_heads     Hq; n_kv_heads Hkv divides Hq; consecutive query heads
 *                 share a KV head
 *   head_dim      d (64 or 128)
 *   n_groups      G >= 1 key groups
 *   group_offsets host [G+1], prefix offsets into group_heads (0 ... Hkv)
 *   group_heads   host [Hkv], the KV heads of each group in the column-block
 *                 order of B_g; together a permutation of 0 .. Hkv-1
 *   ranks         host [G], r_g >= 16, a multiple of 16
 *   rank_v        r_v >= 16, a multiple of 16
 *   dtype         element type of q, caches, factors, x and out
 * R_k = sum_g r_g.  Key latent of group g occupies columns
 * [sum_{g'<g} r_g', +r_g) of a key-cache row.
 */
typedef struct {
  int32_t hidden;
  int32_t n_q_heads;
  int32_t n_kv_heads;
  int32_t head_dim;
  int32_t n_groups;
  const int32_t* group_offsets;
  const int32_t* group_heads;
  const int32_t* ranks;
  int32_t rank_v;
  int32_t dtype; /* dck_dtype */
} dck_layer_desc;

/* Text of a status code (static storage). */
const char* dck_status_string(int32_t status);

/* Checks a descriptor without launching anything. */
dck_status dck_validate_desc(const dck_layer_desc* desc);

/*
 * Latent append (Sec. III-A z = x L; Sec. III-C L_g; Sec. III-D L_v).
 *   x       [n_tok, D] new tokens' hidden states
 *   A_k     [D, R_k] the key down-factors A_g side by side in group order
 *   A_v     [D, r_v]
 *   d_rows  device int64 [n_tok]: cache row that receives token i
 *   kcache  [n_rows, R_k]  <- row d_rows[i] = x_i A_k   (rounded to dtype)
 *   vcache  [n_rows, r_v]  <- row d_rows[i] = x_i A_v
 * Accumulation is fp32.  Rows outside [0, n_rows) are skipped and recorded
 * as a device error.  n_tok = 0 is a no-op.  The workspace (size from
 * dck_latent_append_workspace_size, may be 0) is scratch owned by the caller.
 */
size_t dck_latent_append_workspace_size(const dck_layer_desc* desc, int32_t n_tok);
dck_status dck_latent_append(const dck_layer_desc* desc, const void* x, int32_t n_tok,
                             const void* A_k, const void* A_v, const int64_t* d_rows,
                             void* kcache, void* vcache, int64_t n_rows,
                             void* workspace, size_t ws_bytes, void* stream);

/*
 * Decode attention over the latent caches (formula at the top of this file).
 *   q           [B, Hq, d] queries before RoPE
 *   kcache      [n_rows, R_k] key latents; vcache [n_rows, r_v] value latents
 *   B_k         packed key up-factors: group g's block B_g [r_g, n_g*d]
 *               (row-major) at element offset sum_{g'<g} r_g' n_g' d
 *   B_v         [r_v, Hkv*d]
 *   d_seq_start device int64 [B]: first cache row of sequence b
 *   d_seq_len   device int32 [B]: L_b; rows d_seq_start[b] .. +L_b-1 are
 *               sequence b's tokens at positions 0 .. L_b-1.  L_b = 0 gives a
 *               zero output row.
 *   rope_theta  RoPE base theta > 0
 *   out         [B, Hq, d]
 *   workspace   scratch of at least dck_decode_workspace_size(desc, B, n_rows)
 *               bytes, 256-byte aligned; its contents need no initialisation
 * Work is balanced over the device's SMs by 128-token tiles (the bf16
 * tensor-core path splits the tiles left over after an even share of whole
 * tiles per SM further, by groups of heads); the split partials live in the
 * workspace and are merged by a last kernel on the same stream.  The bf16 tensor-core path also keeps per-tile softmax
 * probabilities there, sized for sequences that do not share cache rows:
 * more than ceil(n_rows / 128) + B tiles in all is reported as DCK_ERR_INVALID
 * by dck_last_device_error and leaves `out` undefined.
 */
/* Workspace bytes for a decode call over `batch` sequences in caches of
 * `n_rows` rows (0 for an invalid descriptor or when the device cannot be
 * queried). */
size_t dck_decode_workspace_size(const dck_layer_desc* desc, int32_t batch, int64_t n_rows);
dck_status dck_decode_attention(const dck_layer_desc* desc, const void* q,
                                const void* kcache, const void* vcache, int64_t n_rows,
                                const void* B_k, const void* B_v,
                                const int64_t* d_seq_start, const int32_t* d_seq_len,
                                int32_t batch, float rope_theta, void* out,
                                void* workspace, size_t ws_bytes, void* stream);

/*
 * Prefill attention: many new tokens per sequence, each attending causally to
 * its prefix, over the same latent caches (Sec. III-A x W ~ z R, Sec. III-C
 * grouped key factors, Sec. III-D value factor; keys and values are rebuilt
 * as for decode, once per cache row for all of a sequence's queries).  The
 * paper describes neither prefill nor a causal mask; the library's reading:
 * the Q_b new tokens of sequence b are the LAST Q_b rows of its cache (their
 * latents appended before the call), query i (0 <= i < Q_b) sits at position
 * p_i = L_b - Q_b + i, rotated there, and attends to the keys at positions
 * 0 .. p_i:
 *   o_ij = sum_{t <= p_i} softmax_t(<q_ij', k_t'> / sqrt(d)) v_t B_v[:, h*d:(h+1)*d]
 * with k_t', q_ij', h and the RoPE convention of the decode formula above.
 *   q            [B, q_max, Hq, d] queries before RoPE; row i of sequence b is
 *                its i-th new token for i < Q_b (later rows are ignored)
 *   d_q_len      device int32 [B]: Q_b, 0 <= Q_b <= min(L_b, q_max); Q_b = 0
 *                writes nothing for sequence b
 *   q_max        the second dimension of q and out, 1 .. 2^24
 *   max_seq_len  an upper bound on every L_b, 1 .. 2^24 (sizes the launch)
 *   kcache .. d_seq_len, rope_theta: as for dck_decode_attention
 *   out          [B, q_max, Hq, d]; rows i < Q_b of each sequence written
 *   workspace    at least dck_prefill_workspace_size(desc, n_rows) bytes,
 *                256-byte aligned: the rebuilt keys (after RoPE) and values,
 *                [n_rows][Hkv][d] bf16 each, written and then read by the call
 * bf16 only, head_dim 128, Hq / Hkv in {1, 2, 4, 8}, at most 16 key groups
 * (DCK_ERR_UNSUPPORTED otherwise; the workspace size query returns 0).  q
 * and out must be 16-byte aligned; n_rows < 2^31 - 256.  Accumulation is
 * fp32 in the tensor cores' accumulators; probabilities are rounded to bf16
 * before the value product and the softmax denominator sums the rounded
 * values.  A sequence with Q_b < 0, Q_b > L_b, Q_b > q_max, L_b > max_seq_len
 * or rows outside the cache is recorded as a device error (DCK_ERR_INVALID
 * from dck_last_device_error) and all q_max of its output rows are zero.
 * Two launches on `stream`: the reconstruction, then the attention.
 */
size_t dck_prefill_workspace_size(const dck_layer_desc* desc, int64_t n_rows);
dck_status dck_prefill_attention(const dck_layer_desc* desc, const void* q, const int32_t* d_q_len,
                                 int32_t q_max, const void* kcache, const void* vcache, int64_t n_rows,
                                 const void* B_k, const void* B_v, const int64_t* d_seq_start,
                                 const int32_t* d_seq_len, int32_t batch, int32_t max_seq_len,
                                 float rope_theta, void* out, void* workspace, size_t ws_bytes,
                                 void* stream);

/*
 * One decode step of a layer: the latent append of the batch's new tokens
 * (Sec. III-A z = x L) followed by decode attention over the caches that now
 * hold them (the formula at the top of this file).
 *   x           [B, D] the new tokens' hidden states, one per sequence
 *   A_k, A_v    as for dck_latent_append
 *   d_rows      device int64 [B]: cache row that receives sequence b's new
 *               token, normally d_seq_start[b] + d_seq_len[b] - 1 (its
 *               position L_b - 1, where its own query attends)
 *   the rest    as for dck_decode_attention; kcache and vcache are written
 *   workspace   at least dck_decode_step_workspace_size(desc, B, n_rows)
 *               bytes, 256-byte aligned
 * On the bf16 tensor-core path with B <= 64 and D a multiple of 128 the
 * append is computed by extra blocks of the call's first kernel (fp32
 * accumulation, one read of A_k and A_v) and the attention kernels read the
 * caches only after it; otherwise the call runs dck_latent_append and then
 * dck_decode_attention on the same stream.  Results equal those of the two
 * calls made one after the other (the appended rows are rounded to the cache
 * dtype in both).  Errors as for the two calls (rows outside the cache are
 * skipped and recorded in the device error word).
 */
size_t dck_decode_step_workspace_size(const dck_layer_desc* desc, int32_t batch, int64_t n_rows);
dck_status dck_decode_step(const dck_layer_desc* desc, const void* x, const void* A_k, const void* A_v,
                           const int64_t* d_rows, const void* q, void* kcache, void* vcache, int64_t n_rows,
                           const void* B_k, const void* B_v, const int64_t* d_seq_start,
                           const int32_t* d_seq_len, int32_t batch, float rope_theta, void* out,
                           void* workspace, size_t ws_bytes, void* stream);

/*
 * Decode attention for callers that cannot allocate device memory (the paper
 * has no counterpart: this is a deployment convenience of the library).
 * A runtime whose device memory is fully reserved by its own pool, a plug-in
 * handed only its input and output tensors, or a loop that must not allocate
 * after start-up cannot provide the workspace of dck_decode_attention.  This
 * entry point computes exactly what dck_decode_attention computes, with the
 * same arguments minus the workspace: the split partials go to a fixed
 * 32 MiB array in the library's own device memory, which every GPU that
 * loads the library holds until the process exits.
 *   - Requests whose dck_decode_workspace_size(desc, B, n_rows) exceeds 32 MiB are rejected
 *     with DCK_ERR_WORKSPACE before anything is launched.
 *   - The first call on a device looks up the array's device address (a
 *     host-side set-up step); make that first call before any stream capture.
 *   - All calls share the one array and it keeps the last call's contents (it
 *     needs no clearing: every value read is written first by the same call).
 *     Calls that overlap on the same GPU (for example on two streams) race on
 *     it: serialise them.  Each GPU has its own copy of the array.
 *   - No device memory is allocated or freed by this call.
 */
dck_status dck_decode_attention_noalloc(const dck_layer_desc* desc, const void* q,
                                        const void* kcache, const void* vcache, int64_t n_rows,
                                        const void* B_k, const void* B_v,
                                        const int64_t* d_seq_start, const int32_t* d_seq_len,
                                        int32_t batch, float rope_theta, void* out, void* stream);

/*
 * Synchronises `stream`, then returns and clears the device error word of the
 * current device: DCK_OK, DCK_ERR_INVALID (a length or row was outside the
 * cache) or DCK_ERR_TIMEOUT (a bounded wait inside a kernel gave up).
 */
dck_status dck_last_device_error(void* stream);

/*
 * Test and measurement hooks.  Each acts only on later calls made by the
 * calling thread (the settings are per thread), so concurrent callers on
 * other threads and streams never see them.
 *
 * dck_set_decode_kernel - kernel selection of the decode path:
 *   0 = automatic (tensor-core kernels where supported, else the CUDA-core kernel)
 *   1 = CUDA-core kernel only
 * Returns this thread's previous value.
 */
int32_t dck_set_decode_kernel(int32_t which);

/*
 * dck_set_timing_events - timing hook of dck_decode_attention: `events` holds
 * n CUDA events (cudaEvent_t, owned by the caller, 2 <= n <= 16).  Each later
 * decode call records events[0] on its stream before its first kernel,
 * events[k] after its k-th kernel for k < n - 1 (k = 1, 2, ...) and
 * events[n - 1] after its last kernel: n = 2 brackets the whole call with
 * nothing recorded between its kernels, n = (kernels + 1) brackets every
 * kernel.  Recording events between kernels delays a kernel that would
 * otherwise start early (programmatic dependent launch), so per-kernel
 * brackets are for a breakdown, not for timing the call.  n = 0 switches the
 * hook off (events is then ignored); any other invalid argument returns
 * DCK_ERR_INVALID.
 */
dck_status dck_set_timing_events(void* const* events, int32_t n);

/* Number of kernels this thread's last decode / append call launched. */
int32_t dck_last_launch_count(void);

/*
 * Self-test of failure detection (not part of the method; the paper has no
 * counterpart): launches on `stream` one block that waits, through the same
 * bounded mbarrier wait every tensor-core kernel uses, on a barrier that
 * nothing arrives at.  After `limit_cycles` SM clock cycles (1000 .. 4e9) the
 * wait gives up, the kernel records a timeout in the device error word and
 * returns, so the next dck_last_device_error reports DCK_ERR_TIMEOUT and the
 * CUDA context stays usable.  Returns DCK_ERR_INVALID for a limit outside that
 * range (nothing is launched), DCK_ERR_CUDA if the launch fails, else DCK_OK.
 */
dck_status dck_selftest_bounded_wait(int64_t limit_cycles, void* stream);

/*
 * Seeded synthetic input (not part of the method): fills n elements of `dst`
 * with the counter-based Gaussian stream `key` starting at element `start`:
 * SplitMix64 draws 2i and 2i+1, the sum of their eight 16-bit fields s,
 * value = float32(2s - 8*65535) * scale (one IEEE fp32 multiply), rounded to
 * bf16 (nearest-even) when dtype is DCK_BF16.  Bit-identical to the Python
 * generator used by the tests.
 */
dck_status dck_synth_gaussian(void* dst, int64_t n, uint64_t key, int64_t start,
                              float scale, int32_t dtype, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* DCK_H_ */
