/*
 * wam_ops.h — kernel-level entry points of the WAMachine library.
 *
 * These expose single hot-path kernels for parity tests and kernel benchmarks.  Every pointer
 * is a device pointer of the current device; nothing is allocated except where noted, and
 * every call is asynchronous on `stream` (a cudaStream_t, NULL = legacy default stream).
 * Return value: 0 on success or a WAM_ERR_* code from wam.h; wam_op_last_error() returns the
 * message of the calling thread's last failure.
 */
#ifndef WAM_OPS_H_
#define WAM_OPS_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* GEMM epilogues (C = A W^T + bias, fused into the accumulator read-back) */
#define WAM_EPI_BF16 0       /* C_bf16[m,n] = acc + bias[n] */
#define WAM_EPI_GELU_BF16 1  /* C_bf16[m,n] = GELU_tanh(acc + bias[n]) (DiT MLP up-projection) */
#define WAM_EPI_RESID_F32 2  /* C_f32[m,n] += gate[item(m), n] * (acc + bias[n]) (adaLN gated
                                residual, item(m) = m / rows_per_item) */
#define WAM_EPI_F32 3        /* C_f32[m,n] = acc + bias[n] */

/*
 * Dense projection of the DiT block (QKV, attention output, MLP up / down):
 *   A  [M, K] bf16 row-major (activations), Wt [N, K] bf16 row-major (weight, K-major),
 *   bias [N] float32 (nullable), gate rows of `gate_stride` floats (RESID only).
 * Runs on the fifth-generation tensor cores (tcgen05.mma, TMEM accumulators, TMA loads).
 * Requires K % 64 == 0, N % 128 == 0, 16-byte aligned pointers.  M >= 1 is arbitrary.
 */
int wam_op_gemm_bf16(const void* A, const void* Wt, const float* bias, void* C, int32_t M,
                     int32_t N, int32_t K, int32_t epilogue, const float* gate,
                     int64_t gate_stride, int32_t rows_per_item, void* stream);

/*
 * The same GEMM with an explicit plan, for tuning and for tests that cover every kernel variant.
 *   tile_n     output tile width: 64, 128 or 256 (0 = the library's choice, as wam_op_gemm_bf16,
 *              with K splitting allowed when a workspace is given)
 *   k_splits   number of K ranges per output tile (0 or 1 = none, up to 4); a split tile's units
 *              publish fp32 partials to `workspace` and the last unit to finish sums them in range
 *              order, so results do not depend on timing.  Needs: the K stages (K / 128 for
 *              64- / 128-wide tiles when K % 128 == 0, else K / 64) divisible by k_splits, and all
 *              tiles x k_splits units in one wave (at most the SM count).
 *   cluster    0 = the library's rule, 1 = single CTAs, 2 = clusters of two CTAs on adjacent
 *              column tiles of the same row block, each loading half of the shared A tile with
 *              TMA multicast into both (64- / 128-wide tiles, an even number of column tiles,
 *              K % 128 == 0, no K split; otherwise single CTAs); 3 = pairs of CTAs (a cluster of
 *              two) running one 256-row MMA (tcgen05 cta_group::2): each CTA loads 128 rows of A and
 *              tile_n / 2 rows of the weight and holds its 128 x tile_n accumulator (tile_n 128 or
 *              256, K % 128 == 0, no K split; WAM_ERR_UNSUPPORTED otherwise).  The accumulation
 *              order over K is the same for every choice.
 *   workspace  device buffer of wam_op_gemm_workspace_bytes() bytes, 16-byte aligned, zero-filled
 *              before its first use (every call leaves it reusable); NULL = no splitting.  Calls
 *              sharing a workspace must be ordered (same stream).
 * Returns WAM_ERR_UNSUPPORTED when the plan does not fit the shape.
 */
int wam_op_gemm_bf16_plan(const void* A, const void* Wt, const float* bias, void* C, int32_t M,
                          int32_t N, int32_t K, int32_t epilogue, const float* gate,
                          int64_t gate_stride, int32_t rows_per_item, int32_t tile_n,
                          int32_t k_splits, int32_t cluster, void* workspace, size_t workspace_bytes,
                          void* stream);

/* Bytes of the split-K workspace of wam_op_gemm_bf16_plan on the current device. */
size_t wam_op_gemm_workspace_bytes(void);

/*
 * The plan the library's shape rule picks for a bf16 projection [M, K] x [K, N] on a GPU with
 * num_sms SMs (what wam_op_gemm_bf16 and the context's projections run): *tile_n = 64, 128 or 256
 * output columns per tile, *cta_pairs = 1 when the tiles run on CTA pairs sharing one two-SM MMA.
 * residual != 0 for a projection whose weight has 64-row boxes and may take 64-wide tiles (the
 * gated-residual projections of a context; every call of wam_op_gemm_bf16).  Host arithmetic
 * only: no device is touched, so it answers on a machine without a GPU.
 * Returns WAM_ERR_INVALID_ARG for M < 1, N or K not multiples of 128 / 64, num_sms < 1 or null
 * outputs.
 */
int wam_op_gemm_plan(int32_t M, int32_t N, int32_t K, int32_t residual, int32_t num_sms, int32_t* tile_n,
                     int32_t* cta_pairs);

/* Same contraction in float32 SIMT (the library's fp32 precision mode). */
int wam_op_gemm_f32(const float* A, const float* Wt, const float* bias, float* C, int32_t M,
                    int32_t N, int32_t K, int32_t epilogue, const float* gate,
                    int64_t gate_stride, int32_t rows_per_item, void* stream);

/*
 * Full bidirectional multi-head attention over the joint token sequence of each item:
 *   qkv [B*N, 3d] (q | k | v column blocks, head h owns columns h*dh .. h*dh+dh-1 of each),
 *   out [B*N, d].  softmax(q k^T / sqrt(dh)) v, no mask.
 * precision WAM_PREC_BF16: bf16 in / out, fp32 accumulation, head dim 64 or 72.
 * precision WAM_PREC_FP32: float32 in / out, any head dim <= 128.
 */
int wam_op_attention(const void* qkv, void* out, int32_t B, int32_t N, int32_t d,
                     int32_t n_heads, int32_t precision, void* stream);

/*
 * adaLN modulate: out[m,:] = LN(h[m,:]) * (1 + scale[item(m),:]) + shift[item(m),:]
 * h [M, d] float32; shift/scale rows of `mod_stride` floats; out bf16 (precision BF16) or f32.
 */
int wam_op_ln_modulate(const float* h, const float* shift, const float* scale,
                       int64_t mod_stride, void* out, int32_t M, int32_t d,
                       int32_t rows_per_item, int32_t precision, void* stream);

/*
 * QKV projection for the tensor-core attention: qkv = A Wt^T + bias with A [M, d], Wt [3d, d]
 * (bf16, K-major), written as bf16 q | k columns into qkv [M, 3d] and with the v columns
 * transposed per item and head into vt [(M / rows_per_item) * d, vt_ld]: element (token n of
 * item i, head h, channel c) at row i*d + h*64 + c, column n.  vt_ld >= rows_per_item, a
 * multiple of 8; columns rows_per_item..vt_ld-1 are never written (keep them zero).  The v
 * columns of qkv are left untouched.
 */
int wam_op_gemm_qkv_vt(const void* A, const void* Wt, const float* bias, void* qkv, void* vt,
                       int32_t M, int32_t d, int32_t rows_per_item, int32_t vt_ld, void* stream);

/*
 * Full bidirectional attention on tcgen05 (head dim dh = d / n_heads, 64 or 72): q and k from
 * qkv [B*N, 3d] (bf16), v from vt as written by wam_op_gemm_qkv_vt with vt_ld = N rounded up to a
 * multiple of 8, out [B*N, d] bf16.  softmax(q k^T / sqrt(dh)) v per item and head, no mask.
 * The head-dim-72 path reads eight V^T rows past each head (the next head's, or nothing past the
 * end of vt); they only feed output columns that are discarded.
 */
int wam_op_attention_tc(const void* qkv, const void* vt, void* out, int32_t B, int32_t N,
                        int32_t d, int32_t n_heads, void* stream);

const char* wam_op_last_error(void);

/*
 * Trajectory Remapping of `batch` finished trajectories that allocates no device memory, for
 * callers that cannot allocate: controllers whose control loop forbids allocation after
 * start-up (bounded step latency), or hosts that own all device memory and hand the library
 * none.  The paper has no counterpart: this is the remap that wam_adapt_state performs on a
 * finished replan, for one executed shift and one (sigma_r, sigma_b0) pair shared by every
 * episode, and it returns the same bits as that remap.
 *   x_bar, x_r, eps, out: [batch, T] float32 device buffers, T = n_video*video_dim +
 *   n_action*action_dim (at most 2^31 - 1); eps may be NULL when shift == 0 and
 *   video_mode == 0 (no slot takes fresh noise then).
 *   normalize != 0 scales each branch's direction to unit RMS; 0 keeps (x_r - x_bar) / sigma_r.
 *   video_mode 0 remaps video without a shift, 1 fills it with sigma_b0 * eps.
 * Scratch: a fixed 64 KiB array inside the library (8192 float64 partial sums) holds the RMS
 * partial sums; batch * 2 * ceil(max(n_video*video_dim, n_action*action_dim) / 2048) must not
 * exceed 8192, else WAM_ERR_UNSUPPORTED.  Every call shares the array and leaves its contents
 * behind; calls that overlap on the GPU race on it and must be serialised by the caller.  The
 * first call on each device looks up the array's address; make it before any stream capture.
 * Errors: WAM_ERR_INVALID_ARG, WAM_ERR_UNSUPPORTED, WAM_ERR_CUDA (message: wam_op_last_error).
 */
int wam_tr_remap_static(const float* x_bar, const float* x_r, const float* eps, float* out,
                        int32_t batch, int32_t n_video, int32_t video_dim, int32_t n_action,
                        int32_t action_dim, int32_t shift, double sigma_r, double sigma_b0,
                        int32_t normalize, int32_t video_mode, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* WAM_OPS_H_ */
