/*
 * map_gb300.h -- C ABI of the GB300 (sm_103a) implementation of MAP's inference-time
 * visual-token pruning path (arxiv 2608.06411, "Learning to Predict Middle-layer
 * Attention in MLLMs for Visual Token Pruning").
 *
 * The path:  (T, V) --map_score--> p_hat --map_select--> keep set --map_gather--> tokens
 *
 * Conventions for every call
 *   - Tensors are plain pointers to row-major, densely packed arrays; bf16 tensors are
 *     passed as void* to 16-bit storage.  Unless a call says otherwise, pointers are
 *     DEVICE pointers owned by the caller and must stay valid until the stream work
 *     completes; map_prune alone also accepts host pointers.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).  Work
 *     is enqueued asynchronously on it; the call returns once enqueued.
 *   - Return value: MAP_OK (0) or a negative MAP_E* code.  Arguments are validated on
 *     the host before anything is enqueued; on an argument error nothing is enqueued.
 *     Device-side failures (a bounded wait that ran out) are recorded in the context
 *     and reported by map_status.
 *   - A context is not thread-safe: one host thread (and one stream at a time) per
 *     context.  Workspace is owned by the context, allocated on first use and grown on
 *     demand (growth synchronises the device).
 */
#ifndef MAP_GB300_H
#define MAP_GB300_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define MAP_OK            0
#define MAP_EINVAL       -1   /* bad argument (null pointer, size, alignment) */
#define MAP_ENOMEM       -2   /* device or host allocation failed */
#define MAP_ECUDA        -3   /* a CUDA runtime / driver call failed */
#define MAP_ETIMEOUT     -4   /* a bounded device-side wait ran out (kernel aborted) */
#define MAP_EUNSUPPORTED -5   /* shape outside what the kernels support (see each call) */
#define MAP_EINTERNAL    -6   /* device-side consistency check failed */

typedef struct map_ctx map_ctx;   /* opaque, owned by the library */

/*
 * Predictor and selection settings.
 *   D, Dh, dp  feature width, predictor MLP width, query/key width d of Eq. 3.
 *              The paper calls the predictor lightweight without giving widths; the
 *              defaults are Dh = 1024, dp = 128 (D = 4096 for LLaVA-NeXT-7B).
 *              Supported: D % 64 == 0, Dh % 256 == 0, dp in {64, 128}.
 *   rope_theta RoPE base (10000); rope_on = 1 applies RoPE to q and k as the paper's
 *              predictor does (section "Cross-Modal Attention Distillation"); 0 turns it
 *              off (used by tests of permutation equivariance).
 *   k0_frac, k0_abs  |R0| (section "Inference-Time Token Pruning"): k0_abs if >= 0,
 *              else floor(k0_frac * K); clamped to [0, K].  The paper does not state
 *              K0; the default is K/2.
 *   lambda     diversity weight: value_i = p_hat_i * rho_i^lambda.  lambda = 1 is Eq. 4;
 *              lambda = 0 reduces the selection to the top-K of p_hat.
 *   tau        a residual with rho_i^2 <= tau * ||v_i||^2 counts as zero (the token is
 *              already in the span); picking such a token keeps it without extending
 *              the basis.  Default 1e-5.
 */
typedef struct {
    int   D, Dh, dp;
    float rope_theta;
    int   rope_on;
    float k0_frac;
    int   k0_abs;
    float lambda;
    float tau;
} map_config;

/* Predictor weights, bf16, PyTorch Linear layout [out, in]; host OR device pointers
 * (map_init copies them).  f_T: wT1 [Dh, D], bT1 [Dh], wT2 [Dh, Dh], bT2 [Dh];
 * W_Q: wQ [dp, Dh]; f_V: wV1, bV1, wV2, bV2 likewise; W_K: wK [dp, Dh]. */
typedef struct {
    const void *wT1, *bT1, *wT2, *bT2, *wQ;
    const void *wV1, *bV1, *wV2, *bV2, *wK;
} map_weights;

/* Fills *cfg with the defaults above (D = 4096, Dh = 1024, dp = 128, theta = 1e4,
 * rope on, K0 = K/2, lambda = 1, tau = 1e-5).  Returns MAP_EINVAL for NULL. */
int map_config_default(map_config *cfg);

/* Creates a context on the current CUDA device, copying the weights (synchronous).
 * Returns MAP_EINVAL for a bad config or NULL pointers, MAP_ENOMEM / MAP_ECUDA on
 * failure (then *out is NULL). */
int map_init(const map_config *cfg, const map_weights *w, map_ctx **out);

/*
 * Predicted attention, Eq. 3 (section "Cross-Modal Attention Distillation"):
 *   p_hat[b, n] = (1/M_b) sum_m softmax_n( <RoPE(W_Q f_T(t_m)), RoPE(W_K f_V(v_n))> / sqrt(dp) )
 * with visual token n at position n and question token m at position N + m.
 *   text_feats  bf16 [sum(lens), D]: the question tokens of all images, packed in
 *               image order (device).
 *   vis_feats   bf16 [B, N, D] (device), 16-byte aligned.
 *   lens        int32 [B] HOST array: question tokens per image, each >= 1.
 *   scores      float32 [B, N] output (device).
 * B >= 1, N >= 1.  Inputs and weights are bf16; every product is accumulated in fp32,
 * and the hidden MLP activations are kept to about 16 significant bits (a bf16 pair)
 * rather than rounded to bf16; q, k, logits and p_hat are fp32.
 */
int map_score(map_ctx *ctx, const void *text_feats, const void *vis_feats,
              const int32_t *lens, int B, int N, float *scores, void *stream);

/*
 * Diversity-aware selection, Eq. 4 (section "Inference-Time Token Pruning"):
 * R0 = top-K0 by p_hat (ties to the lower index), then greedily
 *   i_t = argmax_{i in C} p_hat_i * ||v_i - B B^T v_i||^lambda
 * until k tokens are kept (ties to the lower index).
 *   scores      float32 [B, N] (device), p_hat from map_score (or any non-negative
 *               importance).
 *   vis_feats   bf16 [B, N, D] (device): the embeddings v_i of the diversity term.
 *   keep_idx    int32 [B, k] output (device): kept token indices restored to ascending
 *               original order; they are also the kept tokens' position ids.
 *   pick_order  int32 [B, k] output (device) or NULL: the same tokens in the order they
 *               were retained (R0 in p_hat order first).
 * k == N keeps every token (keep_idx = pick_order = 0..N-1); k == 0 is a no-op;
 * k > N is MAP_EINVAL.  Supported: N <= 16384; k <= 4096 for plain top-k (lambda = 0 or
 * K0 = k), k <= 768 with the diversity term (MAP_EUNSUPPORTED beyond).
 * Asynchronous like the other calls: after its first rounds the selection runs as a
 * device-side loop (a CUDA graph whose WHILE node repeats a round while an image still
 * selects; built on the first call of a shape and workspace, then cached in the context), so
 * the host never waits for it.  A device-side failure (a bounded wait that ran out, or the
 * loop's iteration cap, set at the most rounds the selection can take:
 * k * (ceil(N / 256) + 1) + ceil(k / 128) + 64) is reported by map_status.
 */
int map_select(map_ctx *ctx, const float *scores, const void *vis_feats, int B, int N,
               int k, int32_t *keep_idx, int32_t *pick_order, void *stream);

/*
 * Compaction (last step of section "Inference-Time Token Pruning"):
 *   out[b, j, :] = vis_feats[b, keep_idx[b, j], :]   (a bit copy of bf16 rows)
 * vis_feats [B, N, D], out [B, k, D], keep_idx [B, k] (device).  vis_feats and out
 * must be 16-byte aligned (MAP_EINVAL otherwise).  Indices outside [0, N) are not
 * copied; they set MAP_EINTERNAL for map_status.
 */
int map_gather(map_ctx *ctx, const void *vis_feats, const int32_t *keep_idx, int B, int N,
               int k, void *out, void *stream);

/*
 * Hand-off to the language model (last paragraph of section "Inference-Time Token
 * Pruning"): the kept tokens, restored to their original order, keep their positional
 * indices and are combined with the question tokens.  For image b, whose sequence starts
 * at row o_b = b k + sum_{b' < b} lens[b'] of `seq`:
 *   seq[o_b + j]     = vis_feats[b, keep_idx[b, j]],  pos_ids[o_b + j]     = keep_idx[b, j] + pos_offset
 *   seq[o_b + k + m] = text_feats[t_b + m],           pos_ids[o_b + k + m] = N + m + pos_offset
 * for j < k and m < lens[b], with t_b = sum_{b' < b} lens[b'] (the question follows the
 * whole image, as in map_score).  pos_offset shifts every position (e.g. by the length of
 * a system prompt placed before the image).
 *   vis_feats  bf16 [B, N, D]; keep_idx int32 [B, k] (map_select's output);
 *   text_feats bf16 [sum(lens), D]; lens int32 [B] HOST array, each >= 0;
 *   seq        bf16 [sum_b (k + lens[b]), D] output; pos_ids int32 [same rows] output.
 * Device pointers, caller-owned; vis_feats, text_feats and seq 16-byte aligned (MAP_EINVAL
 * otherwise); 0 <= k <= N.  An index outside [0, N) is not copied: its pos_ids entry is
 * -1 and map_status reports MAP_EINTERNAL.
 */
int map_assemble(map_ctx *ctx, const void *vis_feats, const int32_t *keep_idx,
                 const void *text_feats, const int32_t *lens, int B, int N, int k,
                 int pos_offset, void *seq, int32_t *pos_ids, void *stream);

/*
 * map_select without allocating memory in the call (the paper has no counterpart; this
 * is a deployment variant of map_select).  Same arguments and limits as map_select, and
 * the same exact greedy picks (a near-tie below fp32 resolution may go either way, as
 * between any two fp32 evaluations), but every scratch buffer is carved from one static
 * device array of MAP_NOALLOC_SCRATCH_BYTES, held by each GPU that loads the library
 * until the process exits.  It is for callers that cannot allocate device memory while
 * they prune: code that runs inside another framework's caching pool or under a fixed
 * device-memory budget, where a cudaMalloc would take memory the budget does not have or
 * fail, and serving paths that must not stall on the allocator (cudaMalloc and cudaFree
 * may synchronise the device).  The call makes no cudaMalloc / cudaFree and allocates
 * through no library.
 * Workspace needed, in bytes (each array rounded up to 256): 17 B*N + 16 B*k + 4 B*256
 * + 8 B + small per-image counters, plus, when the diversity term is on (lambda > 0 and
 * K0 < k), 4 B*N*ceil4(k) + 2 B*R*D + 4 B*256*R with R = ceil16(256 + k).  A request
 * that does not fit returns MAP_EUNSUPPORTED and does nothing.  One LLaVA-NeXT image
 * (N = 2880, k = 160, D = 4096) needs about 6 MB.
 * Unlike map_select, whose later rounds run as a device-side loop, it waits on the host
 * for bursts of selection rounds (it synchronises `stream`); a device-side error is
 * returned and also recorded for map_status.  It skips map_select's tensor-core
 * projection pass (every candidate starts from its bound p_hat * ||v||^lambda), so it
 * runs more selection rounds for the same picks.
 * The first call on a device looks the array's address up (device must be current);
 * make that call before any stream capture.  All calls share the array and it keeps the
 * last call's contents; calls whose GPU work overlaps (other streams, other threads)
 * race on it and must be serialised by the caller.
 */
#define MAP_NOALLOC_SCRATCH_BYTES (16u * 1024u * 1024u)
int map_select_noalloc(map_ctx *ctx, const float *scores, const void *vis_feats, int B, int N,
                       int k, int32_t *keep_idx, int32_t *pick_order, void *stream);

/*
 * The whole path in one call: score, select, gather.  Pointers may be HOST or DEVICE
 * memory (detected per pointer); host inputs are copied in and host outputs copied out
 * on `stream`, and the call synchronises `stream` before returning when any pointer is
 * host memory.  text_feats, vis_feats, lens as for map_score (lens is always host);
 * out bf16 [B, k, D]; keep_idx int32 [B, k]; scores float32 [B, N] or NULL.
 */
int map_prune(map_ctx *ctx, const void *text_feats, const void *vis_feats,
              const int32_t *lens, int B, int N, int k, void *out, int32_t *keep_idx,
              float *scores, void *stream);

/*
 * Question Contrastive Teacher Selection (section "Question Contrastive Teacher
 * Selection", Eq. 1 and Eq. 2): the teacher layer whose attention supervises the
 * predictor during training.  For every sample b and language-model layer l:
 *   a^l_n     = 1/(H M_b) sum_h sum_m A^l[h, m, n]                        (Eq. 1)
 *   p^l       = a^l / sum_n a^l_n          (l1 normalisation over visual tokens)
 *   p_ref^l   = the same for the reference question's attention (M_ref tokens)
 *   js[b, l]  = D_JS(p^l, p_ref^l) in nats (natural logarithm)
 *   teacher[b] = l* = argmax_l js[b, l], ties to the lower layer               (Eq. 2)
 * A layer whose aggregate sums to zero (M_b = 0, or attention that is all zero) gets the
 * uniform distribution 1/N.  Context-free: it needs no map_init and no workspace.
 *   attn       bf16, the samples' text-to-vision attention, packed in sample order: sample
 *              b is a dense [L, H, lens[b], N] block (row (h, m) of layer l holds the
 *              attention of question token m to the N visual tokens at head h).  Values
 *              must be finite and non-negative (attention probabilities).
 *   lens       int32 [B] HOST array: question tokens M_b per sample, each >= 0.
 *   attn_ref   bf16 [B, L, H, M_ref, N]: the reference question's attention.
 *   p, p_ref   float32 [B, L, N] outputs: the distributions p^l and p_ref^l.
 *   js         float32 [B, L] output; teacher int32 [B] output (while the call runs it
 *              also counts the finished layers of each sample).
 *   teacher_p  float32 [B, N] output (p^{l*} of each sample) or NULL.
 * All device pointers, caller-owned; attn and attn_ref 2-byte aligned (16-byte alignment
 * with N % 8 == 0 takes the fastest path).  B, L, H, N, M_ref >= 1 (MAP_EINVAL
 * otherwise); L <= 65535.  Asynchronous on `stream`; no device-side error conditions.
 */
int map_qcts(const void *attn, const int32_t *lens, const void *attn_ref, int M_ref, int B,
             int L, int H, int N, float *p, float *p_ref, float *js, int32_t *teacher,
             float *teacher_p, void *stream);

/*
 * Ragged batches (variable-resolution images, e.g. Qwen2.5-VL's dynamic token counts): the
 * same three steps on a padded layout.  vis_feats is [B, N, D] with N the largest token
 * count; image b's visual tokens are rows 0 .. n_valid[b]-1 and the rows after them are
 * padding whose contents are never used.  n_valid int32 [B] is a HOST array with
 * 1 <= n_valid[b] <= N (MAP_EINVAL otherwise).  Per image, the results equal those of the
 * unpadded call on its n_valid[b] tokens: Eq. 3's softmax runs over n < n_valid[b] only and
 * the question follows the image (positions n_valid[b] + m); scores[b, n] = 0 for padding;
 * the selection never retains padding, so k <= min_b n_valid[b] (MAP_EINVAL otherwise).
 * Other arguments, limits and buffer rules as for map_score / map_select / map_prune
 * (map_prune_ragged also accepts host buffers).  The padding rows still pass through the
 * predictor's GEMMs, so the cost is that of the padded batch.
 */
int map_score_ragged(map_ctx *ctx, const void *text_feats, const void *vis_feats,
                     const int32_t *lens, const int32_t *n_valid, int B, int N, float *scores,
                     void *stream);
int map_select_ragged(map_ctx *ctx, const float *scores, const void *vis_feats,
                      const int32_t *n_valid, int B, int N, int k, int32_t *keep_idx,
                      int32_t *pick_order, void *stream);
int map_prune_ragged(map_ctx *ctx, const void *text_feats, const void *vis_feats,
                     const int32_t *lens, const int32_t *n_valid, int B, int N, int k, void *out,
                     int32_t *keep_idx, float *scores, void *stream);
/* map_assemble for a ragged batch: question token m of image b sits at position
 * n_valid[b] + m (+ pos_offset), and kept indices must lie in [0, n_valid[b]). */
int map_assemble_ragged(map_ctx *ctx, const void *vis_feats, const int32_t *keep_idx,
                        const void *text_feats, const int32_t *lens, const int32_t *n_valid,
                        int B, int N, int k, int pos_offset, void *seq, int32_t *pos_ids,
                        void *stream);

/*
 * Predictor distillation step (section "Cross-Modal Attention Distillation"): the predictor
 * is trained offline by minimising D_KL(p^{l*} || p_hat) (the teacher distribution chosen by
 * QCTS, e.g. map_qcts's teacher_p, against Eq. 3's prediction).  This call computes the batch
 * loss  L = (1/B) sum_b sum_n p*_b[n] log(p*_b[n] / p_hat_b[n])  (0 log 0 = 0) with the
 * context's weights and the gradient dL/dW of every predictor weight, through Eq. 3's
 * softmax-mean, RoPE, W_Q / W_K and both MLPs (the second MLP layer and the projection are
 * kept separate here, unlike the inference path).  The optimiser update is the caller's.
 *   text_feats, vis_feats, lens  as for map_score (lens HOST, each >= 1).
 *   teacher    float32 [B, N] (device): each row a distribution over the N visual tokens.
 *   loss       float32 [1] output (device).
 *   grads      float32 device outputs, each with its weight's shape (wT1 [Dh, D], bT1 [Dh],
 *              wT2 [Dh, Dh], bT2 [Dh], wQ [dp, Dh], and the same for V / K); overwritten.
 * fp32 arithmetic throughout (bf16 inputs decoded exactly); deterministic.  Workspace (about
 * 4 (B N + sum(lens)) (D + 5 Dh + 4 dp) + 4 sum(lens) N bytes) is owned by the context.
 * B N <= 2^24 and sum(lens) <= 2^24 (MAP_EUNSUPPORTED beyond).
 */
typedef struct {
    float *wT1, *bT1, *wT2, *bT2, *wQ;
    float *wV1, *bV1, *wV2, *bV2, *wK;
} map_grads;

int map_distill_grad(map_ctx *ctx, const void *text_feats, const void *vis_feats,
                     const int32_t *lens, const float *teacher, int B, int N, float *loss,
                     const map_grads *grads, void *stream);

/* Synchronises `stream` and returns the first deferred device-side error recorded by
 * this context since the last call (MAP_ETIMEOUT, MAP_EINTERNAL), clearing it; else a
 * CUDA error as MAP_ECUDA; else MAP_OK. */
int map_status(map_ctx *ctx, void *stream);

/* Frees the context and its workspace (synchronises the device first).  NULL is a no-op. */
void map_destroy(map_ctx *ctx);

/* Static description of a MAP_E* code. */
const char *map_strerror(int code);

/* ---------------------------------------------------------------- instrumentation
 * Counters and per-kernel CUDA-event timing used by the benchmark; not part of the
 * paper's method. */
typedef struct {
    long long launches;       /* kernels this context has launched */
    long long select_rounds;  /* selection rounds run (one round = choose, Gram, greedy) */
    long long gram_rows;      /* Gram-block rows evaluated by the selection */
} map_counters;

/* The launches of the selection's device-side loop are counted on the device: this call reads
 * that count (a synchronous copy), so it includes the loop iterations that have completed. */
int map_get_counters(map_ctx *ctx, map_counters *out);

/* Kernel ids for timing. */
#define MAP_K_GEMM_FV1    0   /* f_V layer 1: V [B*N, D] x wV1^T, GELU */
#define MAP_K_GEMM_FV2    1   /* no launches: f_V layer 2 is folded into W_K (W_K wV2) */
#define MAP_K_GEMM_WK     2   /* folded W_K wV2 projection with RoPE */
#define MAP_K_GEMM_TEXT   3   /* f_T layer 1 and the folded W_Q wT2 projection together */
#define MAP_K_SCORES      4   /* softmax statistics + mean */
#define MAP_K_SELECT      5   /* everything in map_select */
#define MAP_K_GATHER      6
#define MAP_K_NUM         7

/* enable != 0 records a CUDA event pair around every launch of the kernels above. */
int map_set_timing(map_ctx *ctx, int enable);
/* Synchronises the device; returns the summed event time (ms) and count of kernel `id`
 * since timing was enabled, and resets them. */
int map_read_timing(map_ctx *ctx, int id, double *total_ms, long long *count);

/* ---------------------------------------------------------------- diagnostics
 * Entry points that expose internal stages for tests.  Not on the pruning path. */

/* y[M, Nout] = epi(x[M, K] @ w[Nout, K]^T + b) with the library's tcgen05 GEMM.
 * epi: 0 = GELU then bf16, 1 = bf16, 3 = fp32 (bias ignored for 3; b may be NULL).
 * Device pointers; x, w bf16; K % 64 == 0, Nout % 64 == 0. */
int map_linear(map_ctx *ctx, const void *x, const void *w, const void *b, int M, int K,
               int Nout, int epi, void *y, void *stream);

/* Limit, in ns, of every wait inside the tensor-core GEMM kernels that this context launches
 * (ns <= 0 restores the default of 2 s).  A wait that runs out makes the kernel stop issuing
 * work, let the copies and MMAs already in flight land, release its tensor memory and exit;
 * map_status then reports MAP_ETIMEOUT.  For tests of that path; MAP_EINVAL for NULL. */
int map_set_wait_limit(map_ctx *ctx, long long ns);

/* map_score that also writes q [sum(lens), dp] and k [B*N, dp] (fp32, after RoPE). */
int map_score_debug(map_ctx *ctx, const void *text_feats, const void *vis_feats,
                    const int32_t *lens, int B, int N, float *scores, float *q_out,
                    float *k_out, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* MAP_GB300_H */
