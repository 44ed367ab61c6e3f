/*
 * jpi.h — C-ABI of the GB300 (sm_103a) action-expert denoise library.
 *
 * The library runs the flow-matching denoise of a pi0.5-style action expert on one GPU: a
 * Gemma-shaped suffix transformer (adaptive RMSNorm conditioned on the flow time, one KV head
 * shared by all query heads, GeGLU MLP) is evaluated once per Euler step, attending over the
 * per-layer KV cache of the VLM prefix plus the suffix tokens' own keys and values, and the
 * action chunk is integrated as x <- x + delta * v over a fixed number of steps.
 *
 * Paper passages this interface follows:
 *   - App. A ("Model Architecture of pi series Models"): the expert's queries come from the
 *     action-noise tokens; its keys/values are the matching LLM layer's KV cache concatenated
 *     with the action tokens; flow matching refines the noise over a fixed number of steps.
 *   - Tab. "Model architecture parameters of pi series VLA models": 18 layers, width 1024,
 *     8 heads x 256, 10 denoising steps.
 *   - Sec. 4.3 "System Design": fixed token length (so one captured CUDA graph is reused),
 *     fixed GPU-resident buffers between components, and all denoising iterations unrolled
 *     into one graph.
 *
 * Conventions for every call:
 *   - Every entry point returns a jpi_status. None aborts, traps or exits. Argument and shape
 *     checks run on the host before anything is enqueued; a failed check enqueues nothing.
 *   - CUDA errors map to JPI_ERR_CUDA. jpi_last_error() returns the calling thread's last
 *     message (valid until that thread's next call into the library).
 *   - Matrices are row-major [out][in] (the nn.Linear layout). Activations are fp32.
 *   - "device pointer" means memory of the GPU that was current when the handle was created.
 *   - A handle is not thread-safe: use it from one host thread and one stream at a time.
 *   - `stream` is a cudaStream_t passed as void* (NULL = the legacy default stream).
 */
#ifndef JPI_H
#define JPI_H

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define JPI_API __attribute__((visibility("default")))
#else
#define JPI_API
#endif

typedef struct jpi_handle jpi_handle;

typedef enum jpi_status {
    JPI_OK = 0,
    JPI_ERR_INVALID_ARG = -1,     /* null pointer, non-positive size, unknown enum value      */
    JPI_ERR_SHAPE = -2,           /* a size outside the handle's configured maxima            */
    JPI_ERR_OOM = -3,             /* device or pinned host allocation failed                  */
    JPI_ERR_CUDA = -4,            /* a CUDA runtime/driver call failed (message in last_error) */
    JPI_ERR_NOT_READY = -5,       /* jpi_denoise before any prefix KV was set                  */
    JPI_ERR_DEVICE_TIMEOUT = -6,  /* a bounded device-side wait gave up (see jpi_device_status) */
    JPI_ERR_UNSUPPORTED = -7      /* a model shape this build's kernels do not cover           */
} jpi_status;

typedef enum jpi_precision {
    JPI_BF16 = 0,   /* bf16 weights and prefix KV, bf16 tensor-core inputs, fp32 accumulation,
                       fp32 residual stream and softmax                                          */
    JPI_FP32 = 1    /* fp32 weights and activations everywhere (verification mode, CUDA cores)   */
} jpi_precision;

/* Most correction items (context tokens, see jpi_set_correction) one request may carry. */
#define JPI_MAX_CORRECTION 8

/* Model dimensions and the handle's maxima. The expert has exactly one KV head. */
typedef struct jpi_config {
    int n_layers;     /* L, number of expert layers (18 for pi0.5)                               */
    int width;        /* W, residual width (1024)                                                */
    int n_heads;      /* H, query heads (8)                                                       */
    int head_dim;     /* D, per-head dimension, also the KV width (256)                           */
    int n_kv_heads;   /* must be 1                                                                */
    int mlp_dim;      /* F, GeGLU hidden size (4096)                                              */
    int action_dim;   /* A, action dimension (32)                                                 */
    int state_dim;    /* S_d, dimension of the continuous state token input (32)                  */
    int time_dim;     /* d_t, sinusoidal time-embedding size (even, >= 4)                         */
    int max_batch;    /* largest batch a call may use                                             */
    int max_prefix;   /* largest prefix length (tokens) of the KV store                           */
    int max_chunk;    /* largest action chunk C; the suffix is 1 + T' + C tokens (state,          */
                      /* T' <= JPI_MAX_CORRECTION correction items, actions)                      */
    int max_steps;    /* largest number of Euler steps per call                                   */
    float rope_base;  /* rotary base for the suffix positions (10000); 0 disables rotary coding   */
    float rms_eps;    /* RMSNorm epsilon (1e-6)                                                   */
    float t_min_period, t_max_period;  /* sinusoidal time-embedding periods (4e-3, 4.0)           */
    jpi_precision precision;
} jpi_config;

/*
 * Expert weights, all fp32, [out][in] row-major. In JPI_BF16 mode the matrices are rounded to
 * bf16 (nearest, ties to even) when packed; biases stay fp32. Per-layer tensors are arrays of
 * n_layers pointers. `on_device` = 1 if every tensor pointer is a device pointer, 0 if host.
 * Shapes (W width, H heads, D head_dim, F mlp_dim, A action_dim, S_d state_dim, d_t time_dim):
 *   state_in_w [W][S_d], state_in_b [W]        action_in_w [W][A], action_in_b [W]
 *   action_out_w [A][W], action_out_b [A]      time_mlp_in_w [W][d_t], time_mlp_in_b [W]
 *   time_mlp_out_w [W][W], time_mlp_out_b [W]  final_mod_w [2W][W], final_mod_b [2W]
 *   per layer: wq [H*D][W], wk [D][W], wv [D][W], wo [W][H*D],
 *              w_gate [F][W], w_up [F][W], w_down [W][F],
 *              attn_mod_w [3W][W], attn_mod_b [3W], mlp_mod_w [3W][W], mlp_mod_b [3W]
 * Modulation rows are ordered (scale sigma, shift beta, gate gamma), each W long; the final
 * modulation has (sigma, beta) only.
 */
typedef struct jpi_weights {
    const float *state_in_w, *state_in_b;
    const float *action_in_w, *action_in_b;
    const float *action_out_w, *action_out_b;
    const float *time_mlp_in_w, *time_mlp_in_b;
    const float *time_mlp_out_w, *time_mlp_out_b;
    const float *final_mod_w, *final_mod_b;
    const float *const *wq, *const *wk, *const *wv, *const *wo;
    const float *const *w_gate, *const *w_up, *const *w_down;
    const float *const *attn_mod_w, *const *attn_mod_b;
    const float *const *mlp_mod_w, *const *mlp_mod_b;
    int on_device;
} jpi_weights;

/*
 * Create a handle: validates `cfg`, allocates every persistent device buffer (sized by the
 * maxima), packs the weights (bf16 rounding, tile layout for the bulk tensor copies) and
 * returns the handle in *out. This is the only call that allocates device memory.
 * Ownership: the weights are copied; the caller may free its buffers when the call returns.
 * Synchronous. Errors: INVALID_ARG (null pointer, bad dims), UNSUPPORTED (dims the kernels
 * do not tile), OOM, CUDA.
 * The environment read here fixes kernel choices for the handle's lifetime:
 * JPI_BATCH_INVARIANT=1 makes every launch choose its kernels and splits as for one request, so
 * a request's actions are identical bit for bit alone and inside any batch (slower from batch 4);
 * JPI_ATTN_SPLITS=n fixes the key splits of the small-batch attention (results agree across
 * split counts to rounding only); JPI_ATTN_T5_MIN_BATCH and JPI_BIG_GEMM_MIN_TOKENS move the
 * batch / token thresholds of the large-batch attention and projection kernels (0 disables them);
 * JPI_ATTN_T5_SPLITS=n fixes the key splits of the large-batch attention (1-4, within one wave of
 * clusters; the same rounding-only agreement); JPI_BIG_SPLIT=n fixes the K split of the large-batch
 * O and down projections (1, 2, 4 or 8).
 */
JPI_API jpi_status jpi_expert_create(const jpi_config* cfg, const jpi_weights* w, jpi_handle** out);

/* Free every resource of the handle (synchronises the device first). NULL is accepted. */
JPI_API jpi_status jpi_expert_destroy(jpi_handle* h);

/*
 * Copy the VLM prefix KV cache into the handle's GPU-resident KV store (App. A: per-layer
 * KV handoff from the LLM to the expert; Sec. 4.3: GPU-resident intermediate buffer).
 *   k_layers[l], v_layers[l]: device pointers, l < n_layers, each [batch][prefix_len][D]
 *                             row-major, fp32 if kv_is_fp32 else bf16 (uint16 bit patterns).
 *   batch <= max_batch, 1 <= prefix_len <= max_prefix. Keys are used as given (already
 *   position-encoded by their producer).
 * Asynchronous on `stream`: the caller keeps its buffers alive until the stream reaches this
 * point. In JPI_BF16 mode fp32 input is rounded to bf16; bf16 input in JPI_FP32 mode is widened.
 * The prefix length fixes the graph shape of later jpi_denoise calls (Sec. 4.3, fixed length).
 */
JPI_API jpi_status jpi_set_prefix_kv(jpi_handle* h, const void* const* k_layers,
                                     const void* const* v_layers, int batch, int prefix_len,
                                     int kv_is_fp32, void* stream);

/*
 * Zero-copy producer access to the KV store: returns device pointers to layer `layer`'s K and
 * V store and its layout. Request b's prefix row p, element d lives at
 *   base + b * (*request_stride) + p * D + d      (elements of the store's type)
 * with the store's element type bf16 in JPI_BF16 mode and fp32 in JPI_FP32 mode. After
 * writing rows 0..prefix_len-1 for requests 0..batch-1, call jpi_commit_prefix.
 */
JPI_API jpi_status jpi_prefix_kv_ptr(jpi_handle* h, int layer, void** k, void** v,
                                     long long* request_stride);
JPI_API jpi_status jpi_commit_prefix(jpi_handle* h, int batch, int prefix_len);

/*
 * Correction items (Sec. 4.1 "Foresight-Aligned Asynchronous Correction", App. B, App. C Alg. 1):
 * the future correction module's prediction of the compressed VLM final-layer state at
 * t + Delta, T' tokens of width d_AE, is given to the action expert as future environment
 * information. The expert takes them as context tokens right after the state token: their
 * rows of the residual stream start as the items themselves (d_AE equals the expert's
 * width, so no projection), the state and context rows see the prefix and each other, and
 * the action rows see every key. The paper does not spell out this wiring; this is the
 * reading the library implements.
 *   items:     device fp32 [batch][num_items][width]
 *   num_items: 0 (no items: the plain expert) .. JPI_MAX_CORRECTION
 *   batch:     1 .. max_batch; later jpi_denoise / jpi_expert_forward calls with items set
 *              must use this batch.
 * The items are copied into the handle on `stream` (the caller may reuse its buffer once the
 * stream reaches this point) and stay until the next call. num_items is part of the graph
 * shape: the first denoise after a change of num_items captures a new graph; new item values
 * with the same count reuse it. Errors: INVALID_ARG, SHAPE, CUDA.
 */
JPI_API jpi_status jpi_set_correction(jpi_handle* h, const float* items, int batch, int num_items,
                                      void* stream);

/*
 * Flow-matching denoise (App. A): x_0 = noise; for k = 0..N-1, t_k = k/N,
 * x_{k+1} = x_k + (1/N) * v(x_k, state, t_k; prefix KV); out_actions = x_N.
 *   state:       device fp32 [batch][S_d]
 *   noise:       device fp32 [batch][chunk][A]
 *   out_actions: device fp32 [batch][chunk][A] (may alias noise)
 *   batch must equal the batch of the last jpi_set_prefix_kv/jpi_commit_prefix (and of the
 *   last jpi_set_correction while items are set); 1 <= chunk <= max_chunk;
 *   1 <= num_steps <= max_steps.
 * The first call for a (batch, chunk, num_steps, prefix_len, num_items) shape captures the whole
 * unrolled N-step loop as one CUDA graph (Sec. 4.3: graph reuse and flow unrolling) and every
 * later call with that shape replays it. Asynchronous on `stream`; inputs are read and the
 * output written in stream order. Errors: INVALID_ARG, SHAPE, NOT_READY, CUDA.
 */
JPI_API jpi_status jpi_denoise(jpi_handle* h, const float* state, const float* noise, int batch,
                               int chunk, int num_steps, float* out_actions, void* stream);

/*
 * The same denoise with HOST buffers: copies state and noise host->device, runs the graph,
 * copies the actions device->host and synchronises `stream` before returning. Pinned host
 * memory gives the fastest copies; pageable memory works. Same shapes and errors as
 * jpi_denoise.
 */
JPI_API jpi_status jpi_denoise_host(jpi_handle* h, const float* state, const float* noise,
                                    int batch, int chunk, int num_steps, float* out_actions,
                                    void* stream);

/*
 * One expert evaluation (one Euler step's velocity) at flow time t, for testing:
 *   x_t [batch][chunk][A] device fp32 in; out_v [batch][chunk][A] device fp32 out;
 *   out_h, if not NULL, receives the residual stream after the last layer,
 *   [batch][1 + T' + chunk][W] fp32 (row 0 of each request is the state token, rows 1..T'
 *   the correction items' context tokens).
 * Not captured in a graph. Asynchronous on `stream`.
 */
JPI_API jpi_status jpi_expert_forward(jpi_handle* h, const float* state, const float* x_t,
                                      float t, int batch, int chunk, float* out_v, float* out_h,
                                      void* stream);

/*
 * jpi_expert_forward without allocation of its own, for callers that cannot call cudaMalloc
 * (code that runs inside a stream capture, or under an allocator that owns all device memory
 * once start-up is over). Same arguments, results and errors as jpi_expert_forward.
 * The paper has no counterpart; this is a deployment convenience.
 *   - It allocates nothing: no cudaMalloc, cudaFree or allocating library routine. The scratch
 *     of its time-conditioning stage (sinusoidal embedding, time-MLP hidden layer, conditioning
 *     vector; 96 KiB) is a fixed device array in the library, which every GPU that loads the
 *     library holds until the process exits. width and time_dim above 8192 return
 *     JPI_ERR_SHAPE. The rest of the evaluation uses the handle's buffers, as
 *     jpi_expert_forward does.
 *   - The calling thread's current device must be the handle's device (else
 *     JPI_ERR_INVALID_ARG). The first call in a CUDA context of a device resolves the array's
 *     device address there (cudaGetSymbolAddress) and keeps it for that context; a new context
 *     on the device (after cudaDeviceReset) resolves it again. Make the first call on a device,
 *     and the first after a reset, before any stream capture on that device. The lookup is
 *     safe to make from several host threads at once.
 *   - Every call shares the one array and overwrites it in full: calls that overlap on the GPU
 *     (on different streams, or with different handles) race on it.
 */
JPI_API jpi_status jpi_expert_forward_noalloc(jpi_handle* h, const float* state, const float* x_t,
                                              float t, int batch, int chunk, float* out_v,
                                              float* out_h, void* stream);

/*
 * Synchronise the handle's device work and report device-side errors: JPI_OK, or
 * JPI_ERR_DEVICE_TIMEOUT if a bounded wait inside a kernel gave up (the kernel then skipped
 * its work and returned; outputs of that call are invalid), or JPI_ERR_CUDA.
 */
JPI_API jpi_status jpi_device_status(jpi_handle* h);

/*
 * Measurement hooks.
 * jpi_graph_kernel_count: number of kernel launches in the captured denoise graph of this
 *   (batch, chunk, num_steps) shape at the current prefix length (captures it if needed).
 * jpi_profile_op: enqueues `reps` back-to-back launches of the kernel(s) of one sub-step, for
 *   timing them alone with events on `stream`. Ops: 0 time conditioning (all num_steps step
 *   times), 1 token embedding, 2 norm + QKV projection + rotary of layer `layer`,
 *   3 attention, 4 output projection + gated residual, 5 norm + gate/up + GeGLU,
 *   6 down projection + gated residual, 7 final norm + action-out + Euler update.
 *   Needs a prefix set with this batch; reads and writes the handle's activation buffers
 *   (their contents are meaningless afterwards until the next jpi_denoise).
 */
JPI_API jpi_status jpi_graph_kernel_count(jpi_handle* h, int batch, int chunk, int num_steps,
                                          int* count);
JPI_API jpi_status jpi_profile_op(jpi_handle* h, int op, int layer, int batch, int chunk,
                                  int num_steps, int reps, void* stream);

/* Bytes of device memory the handle holds (weights, KV store, activations, workspaces). */
JPI_API jpi_status jpi_memory_usage(const jpi_handle* h, long long* bytes);

/* Thread-local message of the calling thread's last failed call ("" if none). */
JPI_API const char* jpi_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* JPI_H */
