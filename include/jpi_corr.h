/*
 * jpi_corr.h — C-ABI of the future correction module and its Q-Former state compressor.
 *
 * Paper passages this interface follows:
 *   - Sec. 4.1 ("Foresight-Aligned Asynchronous Correction"): the module takes the compressed
 *     final-layer output of the VLM at time t and the actions committed for execution, and
 *     predicts the compressed final-layer output at t + Delta, which the action expert then uses
 *     (jpi_set_correction in jpi.h takes it as correction items). About 40M parameters.
 *   - App. B ("Architecture of Future Correction Module", and the caption of its figure): the
 *     compressor is a Q-Former block producing T' = 4 tokens of width d_AE from the VLM's T
 *     tokens of width d_VLM; the actions pass an MLP and a Transformer block whose last token is
 *     kept; the two branches are joined, projected and passed through two Transformer blocks;
 *     a correction head gives the predicted state and a confidence head one scalar.
 *   - Eq. 2: the confidence is trained toward minus the prediction error, so it is a
 *     non-positive score in distribution; App. C Alg. 1 compares it with a threshold theta < 0.
 * The widths, norms and activations the paper leaves open are fixed as follows (the same
 * readings as the library's CPU reference): every block is pre-LayerNorm (biased variance),
 * attention has biased q/k/v/o projections and every key visible, MLPs are
 * W2 gelu_tanh(W1 x + b1) + b2, the Q-Former's VLM tokens get no norm and no position code,
 * each committed action k adds row k of a learned position table, the action summary is
 * appended feature-wise to each compressed token and projected back to d_AE, and the
 * confidence is a linear map of the mean of the head's normalised tokens.
 *
 * Conventions are those of jpi.h: every entry point returns a jpi_status, checks its
 * arguments on the host before anything is enqueued, never aborts, and leaves its message in
 * jpi_last_error(). Matrices are row-major [out][in]; activations are fp32; "device pointer"
 * means memory of the GPU that was current at create time; a handle is used from one host
 * thread and one stream at a time.
 */
#ifndef JPI_CORR_H
#define JPI_CORR_H

#include "jpi.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct jpi_corr_handle jpi_corr_handle;

/* Largest number of committed actions one call may pass. */
#define JPI_CORR_MAX_DELTA 64

typedef struct jpi_corr_config {
    int width;           /* d_AE, the module's width = the action expert's width; a multiple of 32 */
    int n_heads;         /* heads of every attention in the module                                  */
    int head_dim;        /* width = n_heads * head_dim; a multiple of 32, at most 256               */
    int mlp_dim;         /* hidden size of every block's MLP                                        */
    int d_vlm;           /* width of the VLM final-layer output the compressor reads                */
    int n_items;         /* T', compressed tokens: 1 .. JPI_MAX_CORRECTION; n_heads * T' <= 64      */
    int action_dim;      /* A                                                                       */
    int max_delta;       /* rows of the position table = most committed actions per call,           */
                         /* 1 .. JPI_CORR_MAX_DELTA                                                 */
    int n_joint;         /* Transformer blocks after the join (2 in App. B), 0 .. 8                 */
    int max_batch;       /* most requests per call                                                  */
    int max_vlm_tokens;  /* most VLM tokens T per compress call                                     */
    float ln_eps;        /* LayerNorm epsilon (1e-6)                                                */
    jpi_precision precision;  /* JPI_BF16: weights stored as bf16 (rounded to nearest even);      */
                              /* JPI_FP32: fp32 weights. Activations and sums are fp32 either way. */
} jpi_corr_config;

/* One pre-LayerNorm Transformer block of width d: x += attn(LN1 x); x += MLP(LN2 x).
 * wq, wk, wv, wo: [d][d]; w1: [mlp_dim][d]; w2: [d][mlp_dim]; vectors [d] (b1: [mlp_dim]). */
typedef struct jpi_corr_block {
    const float *ln1_w, *ln1_b, *wq, *bq, *wk, *bk, *wv, *bv, *wo, *bo;
    const float *ln2_w, *ln2_b, *w1, *b1, *w2, *b2;
} jpi_corr_block;

/* All weights, fp32, host or device pointers (on_device selects which); create copies them. */
typedef struct jpi_corr_weights {
    /* Q-Former compressor. qf_sa is its query self-attention (its ln2/mlp fields are unused and
     * may be NULL); qf_ca_* the cross-attention into the VLM output (wk, wv: [d][d_vlm]);
     * qf_ln2 normalises the queries before it, qf_ln3 before the MLP, qf_lnf the output. */
    const float* qf_query;                      /* [T'][d] learned queries                        */
    jpi_corr_block qf_sa;
    const float *qf_ln2_w, *qf_ln2_b;
    const float *qf_ca_wq, *qf_ca_bq, *qf_ca_wk, *qf_ca_bk, *qf_ca_wv, *qf_ca_bv, *qf_ca_wo, *qf_ca_bo;
    const float *qf_ln3_w, *qf_ln3_b, *qf_mlp_w1, *qf_mlp_b1, *qf_mlp_w2, *qf_mlp_b2;
    const float *qf_lnf_w, *qf_lnf_b;
    /* Action branch: gelu_tanh(a W1^T + b1) W2^T + b2 + pos[k], then block ab. */
    const float *act_w1, *act_b1;               /* [d][A], [d]                                    */
    const float *act_w2, *act_b2;               /* [d][d], [d]                                    */
    const float* act_pos;                       /* [max_delta][d]                                 */
    jpi_corr_block ab;
    /* Join, joint blocks and heads. */
    const float *fuse_w, *fuse_b;               /* [d][2d] over [compressed token ; summary], [d] */
    const jpi_corr_block* jb;                   /* n_joint blocks                                 */
    const float *head_ln_w, *head_ln_b;
    const float *corr_w, *corr_b;               /* [d][d], [d]                                    */
    const float *conf_w, *conf_b;               /* [d] (one row), [1]                             */
    int on_device;
} jpi_corr_weights;

/* Creates a handle: checks the shapes, copies (and for JPI_BF16 rounds) the weights, allocates
 * every buffer for the configured maxima, and evaluates once what depends on the weights alone
 * (the compressor's query self-attention and the cross-attention queries mapped into VLM space).
 * Synchronous; returns after the device work finished. On failure *out is NULL. */
JPI_API jpi_status jpi_corr_create(const jpi_corr_config* cfg, const jpi_corr_weights* w,
                                   jpi_corr_handle** out);
JPI_API jpi_status jpi_corr_destroy(jpi_corr_handle* h);   /* NULL is a no-op */

/* Q-Former compressor (App. B): h_vlm [batch][n_tokens][d_vlm] device, fp32 (vlm_is_fp32 = 1)
 * or bf16 (0), the VLM's final-layer output of each request -> out_state [batch][T'][d] fp32
 * device, the compressed state. 1 <= batch <= max_batch, 1 <= n_tokens <= max_vlm_tokens.
 * Enqueued on `stream`; the inputs must stay valid until the stream reaches the call.
 * The call copies h_vlm into the handle, replays the kernel sequence as a CUDA graph captured the
 * first time this (batch, n_tokens, input type) is asked for (on the handle's own stream, so the
 * first call of a shape should not itself be inside a stream capture), and copies the result to
 * out_state. */
JPI_API jpi_status jpi_corr_compress(jpi_corr_handle* h, const void* h_vlm, int vlm_is_fp32,
                                     int batch, int n_tokens, float* out_state, void* stream);

/* Future correction (App. B, Alg. 1's f_corr): state [batch][T'][d] fp32 device (a compressed
 * state: from jpi_corr_compress, or the previous prediction) and actions [batch][delta][A] fp32
 * device, the committed actions in execution order -> out_state [batch][T'][d] fp32 device, the
 * predicted compressed state at t + delta (ready to pass to jpi_set_correction), and
 * out_confidence [batch] fp32 device (may be NULL). 1 <= delta <= max_delta. out_state may be
 * the same buffer as state. Enqueued on `stream`; like jpi_corr_compress it copies its inputs in,
 * replays a graph captured once per (batch, delta) and copies its outputs out. */
JPI_API jpi_status jpi_corr_predict(jpi_corr_handle* h, const float* state, const float* actions,
                                    int batch, int delta, float* out_state, float* out_confidence,
                                    void* stream);

/* Bytes of device memory the handle holds. */
JPI_API jpi_status jpi_corr_memory_usage(const jpi_corr_handle* h, long long* bytes);

#ifdef __cplusplus
}
#endif

#endif /* JPI_CORR_H */
