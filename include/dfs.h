/*
 * dfs.h - C ABI of the GB300 (sm_103a) engine for step-specific pruned video-DiT blocks
 * ("Dynamic-in-Few-Step": a few-step distilled DiT whose every denoising step keeps its
 * own subset of attention heads and FFN hidden-channel chunks, Sec. 3.2 and Sec. 4.3).
 *
 * Conventions shared by every entry point
 *   - Tensors are row-major.  bf16 means IEEE bfloat16 bit patterns (uint16_t storage).
 *   - Linear weights are [out, in] (so every projection is y = x W^T + b).
 *   - "device" pointers are CUDA global-memory addresses of the current device; "host"
 *     pointers are ordinary CPU memory.  Nothing here takes or returns torch types.
 *   - Every device pointer passed in must be 16-byte aligned (cudaMalloc and torch
 *     allocations are); a misaligned one is rejected with DFS_EINVAL before any GPU work.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).  All GPU
 *     work is enqueued on it; no entry point synchronises except dfs_plan_create,
 *     dfs_plan_sync and dfs_block_forward_host, which say so.
 *   - Errors are returned as dfs_status and never thrown across the ABI; dfs_last_error()
 *     gives a message for the calling thread.  On any error nothing is written to `out`.
 *   - A plan may be used from one host thread at a time.
 *   - CUDA graphs: dfs_block_forward, dfs_block_forward_layer, dfs_denoise,
 *     dfs_model_forward and dfs_model_denoise enqueue only kernel launches and
 *     device-to-device copies, with no allocation and no synchronisation, so a call made
 *     while `stream` is capturing (cudaStreamBeginCapture) is recorded into the graph.
 *     A replay reuses the pointers
 *     and host scalars (timesteps) of the capture and reads the device buffers' contents at
 *     replay time.  Per-kernel profiling (dfs_plan_profile) must be off while capturing.
 */
#ifndef DFS_H_
#define DFS_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct dfs_plan dfs_plan; /* opaque; owned by the library */

typedef enum {
  DFS_OK = 0,
  DFS_EINVAL = 1,        /* bad argument, shape, mask or pointer                      */
  DFS_ENOMEM = 2,        /* device or host allocation failed                          */
  DFS_ECUDA = 3,         /* a CUDA runtime / driver call failed                       */
  DFS_ETIMEOUT = 4,      /* a kernel's bounded wait expired; its results are invalid   */
  DFS_EUNSUPPORTED = 5   /* valid request the library does not implement               */
} dfs_status;

/* How a plan holds the weights of the retained units (Sec. 4.3, Fig. 1(c)).
 *   DFS_ENGINE_COMPACTED: every (step, layer) gets its own dense copy of its retained
 *     weights, gathered once at plan creation; the projections read them as stored.
 *     Weight memory: the sum over steps of the retained weights.
 *   DFS_ENGINE_UNION: the plan keeps one union super-model per layer (the weights of the
 *     units retained at ANY step, theta_union) plus the per-step index tables I_t.  At every
 *     forward the head-granular projections (QKV, output, cross-attention Q / output)
 *     gather the step's heads from the union inside their TMA producer, and the step's FFN
 *     panels (8-channel chunks) are gathered from the union into one plan-owned scratch
 *     pair (sized for the largest step) by the compaction kernel.  Weight memory: the union
 *     plus that scratch.  Results are bit-identical to DFS_ENGINE_COMPACTED (the same
 *     operands reach the tensor cores in the same order). */
typedef enum { DFS_ENGINE_COMPACTED = 0, DFS_ENGINE_UNION = 1 } dfs_engine;

/* Block shapes.  N = grid_t * grid_h * grid_w latent tokens (frame-major).
 *   dim = n_heads * head_dim, head_dim in {64, 128}, ffn_dim % ffn_chunk == 0,
 *   ffn_chunk = 8 (App. A), n_steps = 4 (Sec. 3.1; 1..8 accepted).
 *   qk_norm_mode: 0 = QK RMSNorm over the retained q (k) channels of a token row,
 *                 1 = over each head's head_dim channels.
 *   has_cross = 1 adds text cross-attention over ctx_len context tokens (1..4096).
 *   engine: a dfs_engine value. */
typedef struct {
  int dim, n_heads, head_dim, ffn_dim, ffn_chunk, n_layers, n_steps;
  int grid_t, grid_h, grid_w;
  int ctx_len, has_cross;
  float ln_eps;      /* LayerNorm / RMSNorm epsilon (1e-6)       */
  float rope_theta;  /* 3D RoPE base (1e4)                       */
  int qk_norm_mode;
  int engine;
} dfs_config;

/* One layer's full (unpruned) weights; bf16 DEVICE pointers, borrowed for the duration
 * of dfs_plan_create only (the plan keeps its own compacted copies).
 *   wq, wk, wv, wo [dim, dim]; bq, bk, bv, bo [dim]; gq, gk [dim] (QK RMSNorm scales);
 *   w_up [ffn_dim, dim]; b_up [ffn_dim]; w_down [dim, ffn_dim]; b_down [dim];
 *   e_mod [6, dim] per-layer adaLN table (rows shift_a, scale_a, gate_a, shift_f,
 *   scale_f, gate_f).  Cross-attention (only read when has_cross): cwq..cwo [dim, dim],
 *   cbq..cbo, cgq, cgk, cln_w, cln_b [dim]. */
typedef struct {
  const void *wq, *bq, *wk, *bk, *wv, *bv, *wo, *bo, *gq, *gk;
  const void *w_up, *b_up, *w_down, *b_down, *e_mod;
  const void *cwq, *cbq, *cwk, *cbk, *cwv, *cbv, *cwo, *cbo, *cgq, *cgk, *cln_w, *cln_b;
} dfs_layer_weights;

/* Binary gates of Sec. 3.2 (1 = retained), HOST pointers, borrowed during create:
 *   block_gate [n_steps][n_layers], head_gate [n_steps][n_layers][n_heads],
 *   xhead_gate [n_steps][n_layers][n_heads] or NULL (= all cross heads kept),
 *   ffn_gate [n_steps][n_layers][ffn_dim / ffn_chunk].  Values must be 0 or 1. */
typedef struct {
  const uint8_t *block_gate, *head_gate, *xhead_gate, *ffn_gate;
} dfs_masks;

/* Builds a plan (Sec. 4.3: the union super-model plus the per-step index tables I_t).
 * Validates every argument on the host before any CUDA call, builds the ascending
 * retained head / chunk lists per (step, layer) and the union lists per layer, gathers
 * the retained weight slices into dense bf16 panels on the device (per (step, layer)
 * under DFS_ENGINE_COMPACTED, per layer from the union under DFS_ENGINE_UNION; one
 * compaction kernel per panel), copies the full bias / modulation vectors, precomputes
 * the RoPE tables and, with has_cross, the context keys / values per (step, layer);
 * allocates the workspace for N tokens.
 *   w_t [6*dim, dim], b_t [6*dim]: shared adaLN linear (bf16 device, borrowed).
 *   ctx [ctx_len, dim] bf16 device or NULL when has_cross == 0 (borrowed).
 * Synchronises `stream` before returning.  On failure *out is NULL and everything
 * allocated so far is freed.  Errors: DFS_EINVAL, DFS_ENOMEM, DFS_ECUDA.
 * Host-side fault injection for tests, read here from the environment: DFS_FAULT_ALLOC=n
 * makes the plan's n-th device allocation fail (DFS_ENOMEM); DFS_FAULT_LAUNCH=n makes the
 * plan's n-th kernel launch (counted over its forwards) be skipped and reported as
 * DFS_ECUDA.  Every kernel launch is wrapped in an NVTX range named "dfs <kind>". */
dfs_status dfs_plan_create(const dfs_config* cfg, const dfs_layer_weights* layers /*[n_layers]*/,
                           const void* w_t, const void* b_t, const dfs_masks* masks,
                           const void* ctx, void* stream, dfs_plan** out);

/* Forward of layer 0 at denoising step `step` (0-based; the paper's t_{step+1}).
 * Defined by Eq. 2 (Sec. 3.2: each gated head / FFN chunk / block output multiplied by
 * its binary gate), the export of the gated network to a dense per-step model (Sec. 3.2)
 * and the per-step index-table engine over the union super-model (Sec. 4.3, Fig. 1(c)):
 * the pruned units are never computed, and the result equals the masked dense block.
 * x, out: [N, dim] bf16 device, caller-owned, must not alias.  t_emb: [dim] bf16
 * device.  Computes, with the step's compacted weights only:
 *   mod = W_t t_emb + b_t + E_l; xm = LN(x)(1+scale_a)+shift_a; qkv = xm Wqkv_s^T + b;
 *   QK RMSNorm + 3D RoPE; attention over the retained heads; x1 = x + gate_a (o Wo_s^T + bo);
 *   [cross-attention]; xm2 = LN(x1)(1+scale_f)+shift_f; h = GELU(xm2 Wup_s^T + bup_s);
 *   out = x1 + gate_f (h Wdown_s^T + b_down).   A block gated off copies x to out.
 * Errors: DFS_EINVAL (null pointer, step/layer out of range, x == out), DFS_ECUDA. */
dfs_status dfs_block_forward(dfs_plan* plan, int step, const void* x, const void* t_emb,
                             void* out, void* stream);

/* As dfs_block_forward for any layer of the plan (same passages: Eq. 2, the Sec. 3.2
 * export, Sec. 4.3; each layer has its own gates and index tables per step). */
dfs_status dfs_block_forward_layer(dfs_plan* plan, int step, int layer, const void* x,
                                   const void* t_emb, void* out, void* stream);

/* End-to-end variant of dfs_block_forward_layer on HOST buffers: copies x [N, dim] and
 * t_emb [dim] (bf16, host; pinned memory gives full copy speed) to plan-owned device
 * staging, runs the forward and copies the result back to `out` (host).  Synchronises
 * `stream` before returning. */
dfs_status dfs_block_forward_host(dfs_plan* plan, int step, int layer, const void* x_host,
                                  const void* t_emb_host, void* out_host, void* stream);

/* Asynchronous variant of dfs_block_forward_host for streaming many host-resident inputs:
 * enqueues the copy of x and t_emb into one of two plan-owned staging slots (on a copy
 * stream of the plan), the forward (on `stream`) and the copy of the result to `out_host`
 * (on a second copy stream), and returns without waiting.  Successive calls alternate the
 * slots, so the input copy of call i+1 and the output copy of call i-1 overlap the forward
 * of call i.  Ordering and ownership:
 *   - out_host holds the result once dfs_plan_sync(plan, stream) has returned (it waits for
 *     the copies of every earlier asynchronous call); until then x_host, t_emb_host and
 *     out_host are in use by the library: the caller must not write x_host / t_emb_host or
 *     read out_host (an out_host of an unsynchronised call is not yet a valid x_host).
 *   - Use one stream for a sequence of calls, as for every forward of a plan.
 *   - The first call allocates the second slot (2 N dim + dim bf16) and creates two streams
 *     and six events, all freed by dfs_plan_destroy.  Pinned host memory (cudaHostAlloc)
 *     is needed for the copies to run asynchronously at full speed.
 * Errors: as dfs_block_forward_layer, plus DFS_ENOMEM on the first call. */
dfs_status dfs_block_forward_host_async(dfs_plan* plan, int step, int layer, const void* x_host,
                                        const void* t_emb_host, void* out_host, void* stream);

/* Allocation-free variant of dfs_block_forward_layer (the paper has no counterpart;
 * this is a deployment convenience).  Same arguments, same kernels in the same order,
 * bit-identical result; the per-call activation workspace lives in a 16 MiB device array
 * that the library declares statically, instead of memory the plan allocated.  For
 * callers that must not allocate device memory while running the model: a host
 * application that owns every device allocation through its own pool and budget, or a
 * latency-critical loop that cannot absorb cudaMalloc's implicit synchronisation.  The
 * plan must already exist, and its device must be the current one (else DFS_EINVAL).
 *   - Nothing is allocated: no cudaMalloc, cudaFree or allocating library routine.  The
 *     TMA descriptors of the workspace operands are encoded on the host at every call
 *     (a few microseconds of CPU time, no device work).
 *   - The first call on a device after a plan was created there looks up the array's
 *     device address (with that device current) and keeps it; make that call before
 *     any stream capture.  dfs_plan_create drops the kept address, because a device
 *     reset (which also invalidates every earlier plan) may move the array.
 *   - Every call on a device shares the one array and leaves its contents behind; no
 *     call relies on what an earlier call left.  Calls whose GPU work overlaps (other
 *     streams, other host threads) race on the array: serialise them.
 *   - Under DFS_ENGINE_UNION the step's FFN panels are still gathered into the plan's
 *     own FFN scratch pair (allocated by dfs_plan_create), as in every forward of that
 *     plan: a call also races with any other forward of the same plan whose GPU work
 *     overlaps it.
 *   - Workspace of a (step, layer), with h = h_s head_dim, c = hc head_dim (cross heads,
 *     0 without cross-attention), f = f_s and every term rounded up to 256 bytes:
 *       24 dim + 2 N dim + 4 N h + 2 h ceil64(N) + 2 N max(h, c) + 4 N dim + 2 N ceil64(f) + 2 N c
 *     bytes; above 16 MiB (16777216 bytes) the call is rejected with DFS_EUNSUPPORTED and
 *     a message giving the need.
 * Errors: as dfs_block_forward_layer, plus DFS_EUNSUPPORTED. */
dfs_status dfs_block_forward_noalloc(dfs_plan* plan, int step, int layer, const void* x,
                                     const void* t_emb, void* out, void* stream);

/* Few-step denoising loop (Sec. 3.1, Fig. 1(b) rollout): for s in 0..n_steps-1, run
 * every layer with its step-s structure (block-gated layers skipped), then
 * latents <- latents + (1/cfg.n_steps) * v with v the last layer's output.
 * latents: [N, dim] bf16 device, in/out.  t_embs: [n_steps, dim] bf16 device. */
dfs_status dfs_denoise(dfs_plan* plan, void* latents, int n_steps, const void* t_embs,
                       void* stream);

/* The Wan-shaped model around the blocks -------------------------------------------
 * (not specified by the paper, which prunes inside the blocks only; the wrapper lets the
 * plan run complete denoising passes on a latent video.)  Readings: patch embedding of a
 * latent video [C, F, H, W] (H = 2 grid_h, W = 2 grid_w, F = grid_t) in patches of
 * 1 x 2 x 2, token n = (f grid_h + y) grid_w + x, feature c*4 + dy*2 + dx; x = patches
 * patch_w^T + patch_b.  Timestep t -> e = [cos(t w_i), sin(t w_i)], w_i = 10000^(-i/(D/2));
 * t_emb = t_w2 SiLU(t_w1 e + t_b1) + t_b2, which feeds every block's modulation (rounded to
 * bf16) and the head.  Head: LN(x) (1 + head_mod[1] + t_emb) + head_mod[0] + t_emb, then
 * v = . head_w^T + head_b, unpatched to [C, F, H, W].  bf16 DEVICE pointers, borrowed
 * during dfs_model_attach only. */
typedef struct {
  int in_channels;                 /* latent channels C (16), even                    */
  int freq_dim;                    /* sinusoid width D (256), multiple of 8, <= 8192   */
  const void *patch_w, *patch_b;   /* [dim, 4 C], [dim]                                */
  const void *t_w1, *t_b1;         /* [dim, D], [dim]                                  */
  const void *t_w2, *t_b2;         /* [dim, dim], [dim]                                */
  const void *head_mod;            /* [2, dim]: shift row, scale row                   */
  const void *head_w, *head_b;     /* [4 C, dim], [4 C]                                */
} dfs_model_weights;

/* Copies the model weights into the plan and allocates the model's buffers (token rows
 * [N, 4 C], the block input [N, dim], the timestep vectors).  May be called again to
 * replace them.  Synchronises `stream`.  Errors: DFS_EINVAL, DFS_ENOMEM, DFS_ECUDA. */
dfs_status dfs_model_attach(dfs_plan* plan, const dfs_model_weights* w, void* stream);

/* One pass of the model at denoising step `step` (its structure) and timestep t (host):
 * latent [C, F, H, W] bf16 device (read), v_out [C, F, H, W] bf16 device (written; may not
 * alias latent).  Errors: DFS_EINVAL (no model attached, bad step, NULL, aliasing),
 * DFS_ECUDA. */
dfs_status dfs_model_forward(dfs_plan* plan, int step, const void* latent, float t, void* v_out, void* stream);

/* Few-step sampling in latent space: for s in 0..n_steps-1, v = model(latent, step s,
 * timesteps[s]) and latent <- latent + (1 / cfg.n_steps) v (block-gated layers skipped).
 * latent [C, F, H, W] bf16 device, in/out; timesteps [n_steps] host floats. */
dfs_status dfs_model_denoise(dfs_plan* plan, void* latent, int n_steps, const float* timesteps, void* stream);

/* Test hooks ---------------------------------------------------------------------- */

/* Index lists of I_t for (step, layer): the per-step index table of Sec. 4.3 / Fig. 1(c),
 * built from the hard gates of Sec. 4.1 (FFN chunks of C = 8 channels, App. A).
 * kind: 0 = retained head ids, 1 = retained FFN
 * chunk ids, 2 = retained cross-attention head ids; 3, 4, 5 = the ids of the layer's
 * union super-model (heads / FFN chunks / cross heads retained at any step of the plan,
 * independent of `step`); 6, 7, 8 = the positions of the step's retained heads / chunks /
 * cross heads inside that union (ascending; kind 3 indexed by kind 6 gives kind 0).
 * Writes *count ids to `out` (host, may be NULL to query the count).  Every engine. */
dfs_status dfs_plan_indices(const dfs_plan* plan, int step, int layer, int kind,
                            int32_t* out, int* count);

/* Device address and shape of a compacted panel: the dense per-step weights of the
 * exported model (Sec. 3.2), i.e. the active parameters of step t gathered through I_t
 * (Sec. 4.3, Fig. 1(c)); bf16, row-major, leading dim *ld in elements.  which: 0 Wqkv [3 h_s dh, dim], 1 bqkv [3 h_s dh], 2 gq [h_s dh],
 * 3 gk [h_s dh], 4 Wo [dim, h_s dh], 5 W_up [f_s, dim], 6 b_up [f_s],
 * 7 W_down [dim, f_s] (leading dim f_s rounded up to a multiple of 64); cross: 8 cWq [hc dh, dim], 9 cbq, 10 cWkv [2 hc dh, dim],
 * 11 cbkv, 12 cgq, 13 cgk, 14 cWo [dim, hc dh].  A panel with zero rows or columns
 * returns *dev == NULL.  Under DFS_ENGINE_UNION the weight matrices (0, 4, 5, 7, 8, 10,
 * 14) have no per-step copy: they return their shape with *dev == NULL. */
dfs_status dfs_plan_panel(const dfs_plan* plan, int step, int layer, int which,
                          const void** dev, int64_t* rows, int64_t* cols, int64_t* ld);

/* Device address and shape of a union panel of `layer` (DFS_ENGINE_UNION only; bf16,
 * row-major, leading dim *ld).  With nu / nf / nx the union head / chunk / cross-head
 * counts: which 0 Wqkv [3 nu dh, dim] (the q, k and v rows of the union heads, in that
 * order), 1 Wo [dim, nu dh], 2 W_up [8 nf, dim], 3 W_down [dim, 8 nf], 4 cWq [nx dh, dim],
 * 5 cWo [dim, nx dh].  Errors:
 * DFS_EINVAL, DFS_EUNSUPPORTED for a plan of another engine. */
dfs_status dfs_plan_union_panel(const dfs_plan* plan, int layer, int which, const void** dev,
                                int64_t* rows, int64_t* cols, int64_t* ld);

/* Device memory held by the plan: *weight_bytes = its weight copies (compacted panels or
 * union panels, with the per-step bias / norm-scale vectors), *device_bytes = every device
 * allocation it owns (weights, workspace including the union engine's FFN scratch,
 * tables).  Host only. */
dfs_status dfs_plan_memory(const dfs_plan* plan, int64_t* weight_bytes, int64_t* device_bytes);

/* Algorithmic FLOPs (2 per multiply-add) of one block forward at (step, layer), closed
 * form over the retained units only: 8 N dim head_dim h_s (QKV and output projections)
 * + 4 N^2 head_dim h_s (Q K^T and P V) + 4 N dim f_s (FFN up and down), plus with
 * cross-attention 4 N dim head_dim hc + 4 ctx_len dim head_dim hc + 4 N ctx_len head_dim hc;
 * 0 for a block gated off.  The ratio to the keep-all value is the per-step FLOP
 * retention that Sec. 5.4 reports (a 24% mean cut for Wan-14B) and Sec. 6 plots. */
dfs_status dfs_plan_flops(const dfs_plan* plan, int step, int layer, double* flops);

/* Workspace buffers left by the last forward on this plan (for intermediate checks):
 * which: 0 xm [N, dim] bf16 (holds xm2 after the FFN norm), 1 qk [N, 2 h_s dh] bf16
 * (q | k after RMSNorm + RoPE), 2 vT [h_s dh, ld] bf16, 3 attn [N, h_s dh] bf16,
 * 4 x1 [N, dim] fp32, 5 h [N, f_s] bf16, 6 mod [6, dim] fp32.  *dtype: 0 bf16, 1 fp32.
 * Shapes refer to the (step, layer) of the last forward. */
dfs_status dfs_plan_workspace(const dfs_plan* plan, int which, void** dev, int64_t* rows,
                              int64_t* cols, int64_t* ld, int* dtype);

/* Waits for `stream` (and for the copies of earlier dfs_block_forward_host_async calls)
 * and reports whether any kernel of this plan hit its bounded wait limit since the last
 * call (DFS_ETIMEOUT) or a CUDA error occurred (DFS_ECUDA).  Clears the plan's device
 * error word. */
dfs_status dfs_plan_sync(dfs_plan* plan, void* stream);

/* Failure-path self test: launches one small kernel on `stream` that waits on a barrier
 * nothing ever completes, through the same bounded wait every pipelined kernel of the
 * library uses.  The wait gives up after about one second, records the timeout in the
 * plan's device error word and returns, so the context stays usable; the next
 * dfs_plan_sync reports DFS_ETIMEOUT (and clears the word).  No fault, trap or hang. */
dfs_status dfs_selftest_wait_timeout(dfs_plan* plan, void* stream);

/* Kernel kinds for dfs_plan_profile_read. */
typedef enum {
  DFS_K_MODULATION = 0,   /* adaLN modulation GEMV (W_t t_emb + b_t + E_l)          */
  DFS_K_ADALN = 1,        /* LayerNorm + modulate (both norms of the block)           */
  DFS_K_GEMM_QKV = 2,     /* QKV projection (bias epilogue, V written transposed)     */
  DFS_K_QK_NORM_ROPE = 3, /* QK RMSNorm + 3D RoPE                                      */
  DFS_K_ATTENTION = 4,    /* self-attention over the retained heads                    */
  DFS_K_GEMM_O = 5,       /* output projection + gated residual                        */
  DFS_K_GEMM_UP = 6,      /* FFN up projection + GELU                                  */
  DFS_K_GEMM_DOWN = 7,    /* FFN down projection + gated residual                      */
  DFS_K_CROSS = 8,        /* every kernel of the cross-attention branch                */
  DFS_K_OTHER = 9,        /* bias-only branches, Euler update, block-gate copies       */
  DFS_K_GATHER = 10,      /* union engine: per-forward FFN panel gathers from the union */
  DFS_K_MODEL = 11,       /* model around the blocks: timestep MLP, patch embed, head   */
  DFS_K_COUNT = 12
} dfs_kernel_kind;

/* Per-kernel timing of the forwards enqueued on this plan.  enable = 1 resets the
 * counters and brackets every later kernel launch with a pair of CUDA events on its
 * stream; enable = 0 stops recording (counters are kept).  Launch counts are kept in
 * both modes.  Host only; no synchronisation. */
dfs_status dfs_plan_profile(dfs_plan* plan, int enable);

/* Sum of the event-measured durations (ms) and the launch count of one kernel kind
 * since the last dfs_plan_profile(plan, 1).  Waits for the recorded events.
 * total_ms is 0 for launches made while recording was off. */
dfs_status dfs_plan_profile_read(dfs_plan* plan, int kind, double* total_ms, int64_t* launches);

/* Soft mask -> hard gate rules of Sec. 4.1, host only (no CUDA call).
 * kind 0 = block: g = (m > 0); kind 1 = head: m holds unit_size entries per head and the
 * head is kept iff their mean (computed in double) is > 0; kind 2 = FFN chunk: one
 * scalar per chunk, g = (m > 0).  m: [n_rows][n_units * unit_size] floats (host),
 * g: [n_rows][n_units] (host). */
dfs_status dfs_gates_from_soft_masks(int kind, int n_rows, int n_units, int unit_size,
                                     const float* m, uint8_t* g);

/* Frees every device and host resource of the plan (NULL is a no-op).  Waits for the
 * plan's outstanding work on the device first. */
void dfs_plan_destroy(dfs_plan* plan);

/* Thread-local message of the last error returned on this thread ("" if none). */
const char* dfs_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* DFS_H_ */
