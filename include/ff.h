/*
 * libff -- Forward-Forward (FF) layer-local training and goodness prediction
 * on one NVIDIA GB300 (sm_103a).
 *
 * The operations follow "Going Forward-Forward in Distributed Deep Learning"
 * (arXiv 2404.08573):
 *   - label overlay ..................... §3 "Negative Data"
 *   - goodness g = sum_j y_j^2, p(real) = sigma(g - theta) ... §3, Eq. 1
 *   - L_i(x), Train(L_i, n), x = [positive; negative] ........ §4
 *   - trainLayer(idx, batch) inside the per-layer loop ........ §4.1, Algorithm 1
 *   - Goodness prediction over all but the first layer ....... §3 "Prediction"
 *   - Adam for the FF layers .................................. §5.1
 * with these readings where the paper is silent: the loss of one pair is
 * softplus(theta - g_pos) + softplus(g_neg - theta), averaged over the pairs;
 * every layer input is normalised to x / max(||x||_2, 1e-12) after the
 * overlay; the overlay replaces features 0..9 with a one-hot of value 1.0;
 * Adam is bias-corrected with eps outside the square root.
 *
 * Conventions that hold for every call:
 *   - Every pointer argument is a DEVICE pointer owned by the caller unless the
 *     call says otherwise; the library never frees caller memory.  A layer
 *     owns its parameters, its Adam moments and its workspace.
 *   - Every call that takes a `stream` (a cudaStream_t, NULL = legacy default
 *     stream) is asynchronous on it.  Argument errors are detected on the host
 *     and returned before anything is enqueued; a failed launch returns
 *     FF_ERR_CUDA.  Errors found by kernels (a bounded wait that timed out, a
 *     non-finite goodness) are latched in the layer and reported by
 *     ff_layer_check().
 *   - A layer must not be used from two streams at the same time.
 *   - Activation buffers (the layer input when no labels are given, h_out)
 *     are row-major in the layer's precision (float for FF_FP32, bfloat16 for
 *     FF_BF16) with a row stride of ff_row_stride(features) elements; the pad
 *     columns are written as zero and never read.
 *   - Raw inputs (the `x` of a call that also takes labels, and of
 *     ff_predict) are dense row-major float32 [rows, in_features].
 *   - Rows 0..B-1 of a train batch are the positive rows, rows B..2B-1 the
 *     negative rows (§4: x is the concatenation of the positive and negative
 *     data).
 *   - No C++ exception crosses this interface.
 */
#ifndef FF_H
#define FF_H

#if defined(__GNUC__)
#define FF_API __attribute__((visibility("default")))
#else
#define FF_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  FF_OK = 0,
  FF_ERR_INVALID_ARG = 1, /* bad pointer, size, shape or precision; nothing enqueued */
  FF_ERR_CUDA = 2,        /* a CUDA runtime/driver call or a launch failed */
  FF_ERR_OOM = 3,         /* device allocation failed */
  FF_ERR_TIMEOUT = 4,     /* a kernel's bounded wait gave up (latched, see ff_layer_check) */
  FF_ERR_NONFINITE = 5,   /* a goodness value was NaN or Inf (latched) */
  FF_ERR_UNSUPPORTED = 6, /* valid request this build or device cannot serve */
  FF_ERR_DEVICE_CHECK = 7 /* a device-side check of the checked build failed (see build.py) */
} ff_status;

typedef enum { FF_FP32 = 0, FF_BF16 = 1 } ff_precision;

typedef struct {
  int in_features;   /* fan-in K  (>= 1; >= 10 when labels are overlaid on this layer) */
  int out_features;  /* fan-out N (>= 1) */
  int has_bias;      /* 1: y = ReLU(x_hat W^T + b); 0: no bias (b stays 0) */
  float theta;       /* goodness threshold of Eq. 1 */
  float lr, beta1, beta2, eps;  /* Adam (§5.1) */
  ff_precision prec; /* FF_FP32: fp32 everywhere. FF_BF16: bf16 GEMM operands,
                        fp32 accumulate, fp32 master weights and moments */
  unsigned long long init_seed; /* W ~ U(+-sqrt(6/K)) from this seed; b = 0 */
  int max_rows;      /* workspace capacity in rows (2B); grows on demand if exceeded */
  int keep_grad;     /* 1: keep dW, db and the operand G of the last train step (ff_layer_get_grad, _operand) */
} ff_layer_config;

typedef struct ff_layer ff_layer; /* opaque */
typedef struct ff_net ff_net;     /* opaque */

/* Human-readable name of a status code (static string, never NULL). */
FF_API const char* ff_status_string(ff_status s);

/* Row stride, in elements, of an activation buffer with `features` columns:
 * features rounded up to a multiple of 8 (16-byte rows for bf16 TMA tiles). */
FF_API int ff_row_stride(int features);

/* Creates one FF layer (§4: the L_i a node trains).  Allocates W [N,K] fp32,
 * b [N], the Adam moments (zero), the bf16 copy of W (FF_BF16) and a
 * workspace for cfg->max_rows rows; initialises W on `stream` from
 * cfg->init_seed with the counter-based SplitMix64 generator (He-uniform).
 * Requires an sm_100-family GPU for FF_BF16 (FF_ERR_UNSUPPORTED otherwise).
 * On success *out owns everything; on error *out is NULL and nothing leaks. */
FF_API ff_status ff_layer_create(const ff_layer_config* cfg, void* stream, ff_layer** out);

/* Waits for the layer's last stream, frees everything it owns.  NULL-safe. */
FF_API ff_status ff_layer_destroy(ff_layer* layer);

/* Label overlay of §3 "Negative Data": out[r, 0..9] = one-hot(labels[r])
 * (value 1.0, replacing the features), out[r, j] = x[r, j] for j >= 10, cast
 * to `prec`; x is dense float32 [rows, features], out an activation buffer
 * [rows, ff_row_stride(features)].  If row_scale is not NULL it receives
 * 1 / max(||out_r||_2, 1e-12) computed in fp32 before the cast.
 * labels should lie in 0..9; a row whose label is outside that range gets
 * an all-zero label area.  features >= 10. */
FF_API ff_status ff_overlay_label(const float* x, const int* labels, int rows, int features,
                           void* out, float* row_scale, ff_precision prec, void* stream);

/* L_i(x) of §4: the layer's forward pass without an update.
 *   x          labels != NULL: raw float32 [rows, in] to overlay (§3);
 *              labels == NULL: activation buffer [rows, ff_row_stride(in)].
 *   row_scale  [rows] 1/||x_r|| of the layer input, or NULL to compute it
 *              (ignored when labels are given: computed by the overlay).
 *   h_out      [rows, ff_row_stride(out)] activation buffer: ReLU(x_hat W^T + b).
 *   next_scale [rows] or NULL: 1 / max(sqrt(g_r), 1e-12), the next layer's
 *              row_scale (||h_r|| = sqrt(g_r)).
 *   goodness   [rows] or NULL: g_r = sum_j h_rj^2 (Eq. 1), from the fp32
 *              accumulator before any rounding of h. */
FF_API ff_status ff_layer_forward(ff_layer* layer, const void* x, const int* labels,
                           const float* row_scale, int rows, void* h_out,
                           float* next_scale, float* goodness, void* stream);

/* trainLayer(idx, batch) of Algorithm 1 / Train(L_i, 1 batch) of §4: one
 * local FF update on the 2B rows of x (B positive then B negative rows).
 * Forward as ff_layer_forward (with the weights before this update), then
 * loss = (1/B) sum_pairs softplus(theta - g_pos) + softplus(g_neg - theta)
 * (the negative log-likelihood of Eq. 1), dL/dz = dL/dg * 2h * [z > 0],
 * dW = dZ^T x_hat, db = sum_rows dZ, and one Adam step on W and b.
 * No gradient leaves the layer.  h_out/next_scale/goodness as in
 * ff_layer_forward (the pre-update forward; the next layer's input);
 * loss [1] or NULL.  B == 0 is a no-op returning FF_OK. */
FF_API ff_status ff_layer_train_step(ff_layer* layer, const void* x, const int* labels,
                              const float* row_scale, int B, void* h_out,
                              float* next_scale, float* goodness, float* loss,
                              void* stream);

/* Goodness prediction of §3 "Prediction": for every label c in 0..9 the raw
 * input x [n, in] (float32) is overlaid with c and run through all layers;
 * the goodness of layers 2..n_layers (layer 1 when n_layers == 1) is summed
 * into goodness[r, c] ([n, 10] float32, or NULL) and pred[r] (int32) is the
 * label with the largest sum, the lowest label on ties.  All layers must share
 * one precision and chain (out_features of layer k == in_features of k+1).
 * Scratch space is owned by layers[0] (grown on demand). n == 0 is a no-op. */
FF_API ff_status ff_predict(ff_layer* const* layers, int n_layers, const float* x, int n,
                     int* pred, float* goodness, void* stream);

/* AdaptiveNEG negative labels of §5: the negative label of a sample is the
 * wrong label the network currently predicts most strongly.  Runs the
 * goodness prediction of ff_predict on x [n, in] (raw float32) and writes
 * neg[r] (int32) = the label c != labels[r] with the largest goodness sum,
 * the lowest such label on ties; goodness [n, 10] (or NULL) as in ff_predict.
 * labels [n] int32 (device) are the true labels; a label outside 0..9 leaves
 * no label out, so neg[r] is then the plain prediction.  Layers, scratch,
 * stream and n == 0 behave as in ff_predict; labels == NULL with n > 0 is
 * FF_ERR_INVALID_ARG. */
FF_API ff_status ff_adaptive_negatives(ff_layer* const* layers, int n_layers, const float* x,
                                       const int* labels, int n, int* neg, float* goodness,
                                       void* stream);

/* ---------------------------------------------------------------------------
 * Softmax prediction head of §3 "Prediction" (Softmax method).  The input,
 * labelled with the neutral label (0.1 in each of the 10 label features),
 * runs once through the layers; the activities of layers 2..L (layer 1 when
 * L == 1), each divided by its own norm max(||h||, 1e-12), form the features
 * A [n, n_features] of a linear softmax layer z = A V^T + c with 10 classes.
 * The head is trained by backpropagation through itself only (mean
 * cross-entropy over the rows, Adam): no gradient reaches the FF layers, which
 * it reads but never changes.  V [10, n_features] and c [10] start at zero.
 * ------------------------------------------------------------------------- */
typedef struct ff_head ff_head;

typedef struct {
  int n_features;    /* sum of out_features of layers 2..L (of layer 1 when L == 1) */
  float lr;          /* Adam learning rate (the paper uses 1e-4 for the softmax layer) */
  float beta1, beta2, eps;
  int max_rows;      /* rows per train step (and per predict chunk); 0 = 4096 */
} ff_head_config;

/* Allocates the head on the current device.  FF_ERR_INVALID_ARG on a bad
 * config, FF_ERR_OOM / FF_ERR_CUDA on allocation failure (nothing leaks). */
FF_API ff_status ff_head_create(const ff_head_config* cfg, ff_head** out);
/* Waits for the head's last stream and frees it.  NULL is a no-op. */
FF_API ff_status ff_head_destroy(ff_head* head);

/* One training step of the head on n (<= max_rows) raw float32 input rows x
 * [n, in_features of layer 1] with true labels [n] int32 (0..9), through
 * layers[0..n_layers-1] (chained, one precision, read only): the neutral
 * forward, logits, softmax, cross-entropy, dV = dz^T A, dc = sum dz and one
 * Adam step on V and c.  loss [1] (device) or NULL receives the mean
 * cross-entropy.  The layers must not be updated concurrently on another
 * stream (order them before `stream`, e.g. with ff_net_sync).  The layer set
 * must match n_features, else FF_ERR_INVALID_ARG. */
FF_API ff_status ff_head_train_step(ff_head* head, ff_layer* const* layers, int n_layers,
                                    const float* x, const int* labels, int n, float* loss,
                                    void* stream);

/* ceil(n / B) consecutive train steps of the head, as ff_head_train_step on
 * rows [tB, tB + B) of x and labels for t = 0, 1, ... (the last step takes the
 * rest), bitwise the same.  The layers do not change during head training,
 * so the neutral forward runs once over many steps' rows (up to 16384 per
 * pass, whole steps) and each step's logits, gradient and Adam update read
 * their rows of the stored activities.  With several passes the next pass's
 * forward runs on a side stream of the head's, into a second workspace,
 * while `stream` runs the current pass's steps.  B <= max_rows; the
 * workspaces grow to the rows of one forward pass.  loss [ceil(n / B)] (device) or NULL receives
 * each step's mean cross-entropy. */
FF_API ff_status ff_head_train_epoch(ff_head* head, ff_layer* const* layers, int n_layers,
                                     const float* x, const int* labels, int n, int B, float* loss,
                                     void* stream);

/* Softmax prediction of n raw input rows (any n; processed in chunks of
 * max_rows): pred [n] int32 = the class with the largest logit (the lowest
 * on ties) and/or logits [n, 10] float32; either may be NULL, not both. */
FF_API ff_status ff_head_predict(ff_head* head, ff_layer* const* layers, int n_layers,
                                 const float* x, int n, int* pred, float* logits, void* stream);

/* Head state to/from host or device buffers (any NULL skipped): V, m_V, v_V
 * [10, n_features]; c, m_c, v_c [10]; the Adam step.  Synchronous. */
FF_API ff_status ff_head_get_state(const ff_head* head, float* V, float* c, float* m_V,
                                   float* v_V, float* m_c, float* v_c, long long* step);
FF_API ff_status ff_head_set_state(ff_head* head, const float* V, const float* c,
                                   const float* m_V, const float* v_V, const float* m_c,
                                   const float* v_c, long long step);
/* The gradient (dV [10, n_features], dc [10]) of the last train step. */
FF_API ff_status ff_head_get_grad(const ff_head* head, float* dV, float* dc);
/* Waits for the head's stream; reports and clears latched device errors
 * (FF_ERR_NONFINITE for non-finite logits or activities). */
FF_API ff_status ff_head_check(ff_head* head);

/* ---------------------------------------------------------------------------
 * Chapter schedule of the pipelined FF algorithms (§4, Algorithms 1 and 2).
 * The E = C * S training epochs are cut into S chapters of C epochs.  In
 * chapter c, layer i trains C epochs over the output of layer i-1 as it
 * stands after that layer's chapter c (layer 1: the raw pairs overlaid with
 * the chapter's labels), then publishes its own output with the updated
 * weights.  Single-Layer PFF runs each layer on its own CUDA stream (one
 * "node" per layer); All-Layers PFF lets `nodes` streams take the chapters in
 * turn, each training all layers.  Both follow the same dependencies and give
 * the same weights bit for bit.  Learning-rate cooldown (§5.1 names one but
 * gives no formula): each layer's lr is constant until epoch
 * cooldown_start * E of its own epochs, then falls linearly to 0 at E.
 * ------------------------------------------------------------------------- */
typedef struct ff_pff ff_pff;

typedef enum { FF_PFF_SINGLE_LAYER = 0, FF_PFF_ALL_LAYERS = 1 } ff_pff_mode;

typedef struct {
  int n_pairs;             /* P: positive/negative pairs in the training set */
  int batch_pairs;         /* pairs per train step (the last batch takes the rest) */
  int epochs_per_chapter;  /* C */
  int chapters;            /* S, chapters of the whole run (E = C * S) */
  ff_pff_mode mode;
  int nodes;               /* FF_PFF_ALL_LAYERS: streams taking chapters in turn (>= 1) */
  float cooldown_start;    /* fraction of E where the lr cooldown starts; >= 1: none */
} ff_pff_config;

/* Binds a chain of layers (one precision, out_features of layer k ==
 * in_features of k+1, layer 1 in_features >= 10) to a schedule: creates its
 * streams and two chapter slots of published output per layer below the top
 * (2P rows each, in HBM), and sizes every layer's workspace for a batch.
 * The layers must outlive the schedule and must not be used elsewhere while
 * a run is in flight. */
FF_API ff_status ff_pff_create(ff_layer* const* layers, int n_layers, const ff_pff_config* cfg,
                               ff_pff** out);
/* Waits for the schedule's streams and frees it (not the layers).  NULL: no-op. */
FF_API ff_status ff_pff_destroy(ff_pff* pff);

/* Enqueues chapters first .. first+count-1 (0-based, within 0..S-1; chapters
 * must be run in order across calls).  x [2P, in_features of layer 1] raw
 * float32 in the batch-major pair layout (batch j: its b positive rows, then
 * the same b images as negative rows); labels [count, 2P] int32, chapter by
 * chapter, in the same row order (the negative rows' labels are the
 * chapter's negative labels: fixed, random or adaptive).  loss [count, L,
 * C * batches] (device) or NULL receives every train step's loss.  Nothing
 * starts before `stream` reaches this call, and `stream` waits for the whole
 * run; the host returns after enqueueing. */
FF_API ff_status ff_pff_run(ff_pff* pff, const float* x, const int* labels, int first, int count,
                            float* loss, void* stream);

/* Host-side bounded wait for everything the schedule has enqueued so far, as
 * ff_net_wait: FF_OK, or FF_ERR_TIMEOUT after timeout_ms milliseconds. */
FF_API ff_status ff_pff_wait(ff_pff* pff, unsigned int timeout_ms);

/* ---------------------------------------------------------------------------
 * Performance-Optimized PFF (§4, "a new goodness function"): each layer has
 * its own softmax block (an ff_head with n_features = the layer's
 * out_features) and the two are trained together by backpropagation through
 * these two layers only, on the block's cross-entropy; there is no negative
 * data.  The block reads the layer's raw activity h: z = h V^T + c.
 * ------------------------------------------------------------------------- */

/* One step on n rows: the layer's forward pass (raw_input != 0: x is raw
 * float32 [n, in_features], overlaid with the neutral label 0.1 in features
 * 0..9; else x is an activation buffer [n, ff_row_stride(in)] with row_scale
 * [n] or NULL as in ff_layer_forward), the block's logits, the mean
 * cross-entropy over labels [n] (int32, 0..9), dV = dz^T h, dc = sum dz,
 * dZ = (dz V) * [h > 0] with the block's weights before this step,
 * dW = dZ^T x_hat, db = sum dZ, then one Adam step of the layer (its own lr)
 * and one of the block (the block's lr).  h_out / next_scale (or NULL) take
 * the activity and the next layer's row scale from the pre-update weights,
 * as in ff_layer_train_step; loss [1] (device) or NULL.  `block` must have
 * n_features == the layer's out_features, else FF_ERR_INVALID_ARG.  The
 * block's Adam step runs on a stream the block owns, beside the layer's
 * weight gradient and Adam; `stream` waits for it before the call's work
 * ends there, so everything is ordered before later work on `stream`. */
FF_API ff_status ff_po_train_step(ff_layer* layer, ff_head* block, const void* x, int raw_input,
                                  const float* row_scale, const int* labels, int n, void* h_out,
                                  float* next_scale, float* loss, void* stream);

/* A Performance-Optimized net on one CUDA stream per layer, as ff_net: layer
 * k and its block (blocks[k], n_features == layers[k] out_features) train
 * batch t while layer k-1 trains batch t+1; bitwise the same as calling
 * ff_po_train_step layer after layer.  max_rows: the largest batch (rows);
 * depth: activation (and label) ring slots.  ff_net_sync, ff_net_wait and
 * ff_net_destroy apply; ff_net_train_step and ff_net_train_step_images do
 * not (FF_ERR_INVALID_ARG). */
FF_API ff_status ff_net_create_po(ff_layer* const* layers, ff_head* const* blocks, int n_layers,
                                  int max_rows, int depth, ff_net** out);
/* One batch: x [rows, in] raw float32 (neutral label on layer 1), labels
 * [rows] int32 (0..9, read by every layer); loss [n_layers] (device) or
 * NULL gets each layer's block cross-entropy.  The caller's stream waits
 * until layer 1 has read x; labels are copied before the call returns on
 * the GPU side of that wait. */
FF_API ff_status ff_net_po_train_step(ff_net* net, const float* x, const int* labels, int rows,
                                      float* loss, void* stream);

/* Prediction of a Performance-Optimized net: the neutral-labelled raw input
 * x [n, in] runs through layers[0..n_layers-1]; pred [n] (int32) is the
 * argmax of the last layer's block (`block`, n_features == the last layer's
 * out_features) on its raw activity, logits [n, 10]; either may be NULL, not
 * both.  Processed in chunks of the block's max_rows. */
FF_API ff_status ff_po_predict(ff_layer* const* layers, int n_layers, ff_head* block, const float* x,
                               int n, int* pred, float* logits, void* stream);

/* Copies the layer state to/from caller buffers, which may be host or device
 * memory: W [N,K] and its Adam moments m_W, v_W [N,K]; b, m_b, v_b [N]; the
 * Adam step counter.  Any pointer may be NULL to skip that tensor.  Both calls
 * first wait for the layer's last stream and are synchronous.  set_state also
 * refreshes the bf16 copy of W. */
FF_API ff_status ff_layer_get_state(const ff_layer* layer, float* W, float* b, float* m_W,
                             float* v_W, float* m_b, float* v_b, long long* step);
FF_API ff_status ff_layer_set_state(ff_layer* layer, const float* W, const float* b,
                             const float* m_W, const float* v_W, const float* m_b,
                             const float* v_b, long long step);

/* Statistics of the last ff_layer_train_step (or ff_net step) of the layer,
 * for logging: stats[0] = mean goodness of the B positive rows, stats[1] =
 * mean goodness of the B negative rows, stats[2] = fraction of the 2B x out
 * activities that are positive (active ReLUs).  Host or device pointer;
 * waits for the layer's last stream.  Zero before the first step. */
FF_API ff_status ff_layer_get_stats(const ff_layer* layer, float* stats);

/* The gradient of the last ff_layer_train_step (dW [N,K], db [N], fp32, host
 * or device pointers; NULL skips).  Needs cfg.keep_grad = 1, else
 * FF_ERR_UNSUPPORTED.  Synchronous. */
FF_API ff_status ff_layer_get_grad(const ff_layer* layer, float* dW, float* db);

/* The weight-gradient operand of the last train step (of ff_layer_train_step
 * or ff_po_train_step): G = diag(s) dZ, the local gradient scaled by each
 * row's input scale, rows [rows, ff_row_stride(out_features)] in the layer's
 * operand type (bf16 in FF_BF16 mode, rounded to nearest even as the
 * weight-gradient GEMM reads it; fp32 otherwise), so that dW = G^T x.
 * rows: the step's rows (2B for a train step, n for a Performance-Optimized
 * step).  Host or device pointer.  Needs cfg.keep_grad = 1 (the operand is
 * otherwise dropped from the cache once read), else FF_ERR_UNSUPPORTED.
 * Synchronous. */
FF_API ff_status ff_layer_get_grad_operand(const ff_layer* layer, void* out, int rows);

/* Waits for the layer's last stream and returns the first latched kernel
 * error (FF_ERR_TIMEOUT, FF_ERR_NONFINITE) or FF_ERR_CUDA, then clears it. */
FF_API ff_status ff_layer_check(ff_layer* layer);

/* Where a bf16 train step forms the rest of the local step of §3 (Eq. 1)
 * after the forward: enable = 1 in the forward GEMM's epilogue -- the CTAs
 * of a row block exchange their goodness partials in a thread-block cluster
 * and write dZ', the bias-gradient and loss partials themselves -- wherever
 * out_features <= 2048; enable = 0 (the default) in a separate kernel after
 * the forward.  Both give bitwise the same results.  The fused form is
 * faster for a layer stepped alone on a stream and slower where several
 * layers' kernels share the GPU (a net on layer streams), since its clusters
 * of up to 8 CTAs need that many free SMs at once.  No effect on fp32
 * layers.  Returns FF_ERR_INVALID_ARG for a NULL layer. */
FF_API ff_status ff_layer_set_fused_local_grad(ff_layer* layer, int enable);

/* A net of layers trained concurrently, one CUDA stream per layer: the
 * single-GPU analogue of Single-Layer PFF (§4.1, Algorithm 1), where node i
 * trains L_i on the output of L_{i-1}.  Here the hand-off is per batch: layer
 * k+1 trains on batch t from layer k's pre-update forward of batch t, while
 * layer k may already train on batch t+1 (inter-stream events, ring buffers
 * of `depth` batches of activations).  The result is bitwise identical to
 * running the same layer steps one after another on one stream.
 * The net borrows the layers (they must outlive it) and owns its streams,
 * events and activation buffers for up to max_B pairs. */
FF_API ff_status ff_net_create(ff_layer* const* layers, int n_layers, int max_B, int depth,
                        ff_net** out);
FF_API ff_status ff_net_destroy(ff_net* net);

/* Enqueues one batch for every layer: x raw float32 [2B, in], labels [2B]
 * (true labels then wrong labels).  `stream` is ordered before layer 1 reads
 * x, and after it finished reading x: the caller may overwrite x once
 * `stream` reaches this point.  loss [n_layers] (device) or NULL receives
 * each layer's loss asynchronously; call ff_net_sync before reading it. */
FF_API ff_status ff_net_train_step(ff_net* net, const float* x, const int* labels, int B,
                            float* loss, void* stream);

/* As ff_net_train_step, with each image sent once per pair: x raw float32
 * [B, in] (the positive and the negative row of pair i share image i, as in
 * §3 "Negative Data"), labels [2B] (true labels then wrong labels).  Layer 1
 * overlays image i with labels[i] for row i and with labels[B + i] for row
 * B + i; the result is bitwise that of ff_net_train_step on x stacked twice.
 * Halves the input bytes a caller copies per step. */
FF_API ff_status ff_net_train_step_images(ff_net* net, const float* x, const int* labels, int B,
                                          float* loss, void* stream);

/* A whole run of batches through the net (§4: layer i trains on the output
 * of layer i-1 computed with that layer's weights before the same step's
 * update; §3 Eq. 1 and §5.1 per layer), in one persistent kernel: the
 * tensor-core tiles of every layer's forward and weight-gradient GEMMs, and
 * the label overlay, local gradient and Adam of every layer, run as tasks
 * on all SMs at once, the layers as a wavefront (layer k on batch t - k: the
 * single-GPU analogue of Single-Layer PFF, Algorithm 1).  Bitwise the same
 * result as ff_net_train_step (or _images) called once per batch.
 *   x: images_per_pair_row = 2: [2 * n_pairs, in] float32 pair batches laid
 *      out as ff_net_train_step takes them, batch t (B pairs, the last one
 *      n_pairs % B) in rows 2tB .. 2tB + 2b (b positive rows, then the same
 *      images again for the negative rows); images_per_pair_row = 1:
 *      [n_pairs, in], one image per pair, as ff_net_train_step_images.
 *   labels: [2 * n_pairs] int32, per batch b true labels then b wrong ones.
 *   loss: [ceil(n_pairs / B), n_layers] (device) or NULL: each batch's loss
 *      per layer.
 * Runs in the persistent kernel when every layer is FF_BF16 with in and out
 * features multiples of 8 (at most 16384 out), at most 8 layers, and 2B a
 * multiple of 256 (at most 16384); the last partial batch, and any net
 * outside these limits, goes through ff_net_train_step.  The first call for
 * a given (B, batch count, layout) builds and keeps a plan (task tables,
 * tensor maps, activation rings; it allocates).  Returns with `stream`
 * ordered after all of it (as ff_net_sync).  Not on a Performance-Optimized
 * net (FF_ERR_INVALID_ARG).
 * Roles: by default every SM runs GEMM tiles and streamed tasks side by side.
 * With the environment variable FF_EPOCH_GEMM_CLUSTERS=n (read when a plan
 * is built; 1 <= n < the number of resident CTA pairs) n pairs run only GEMM
 * tiles and the other CTAs only the streamed tasks -- the same bits, and on
 * the 784-2000x4 epoch slower for every n. */
FF_API ff_status ff_net_train_epoch(ff_net* net, const float* x, const int* labels, int n_pairs, int B,
                                    int images_per_pair_row, float* loss, void* stream);

/* Instrumentation of ff_net_train_epoch (not part of the method).
 * enable = 1 / 0 switches per-task tracing of later epoch calls on or off
 * (-1 leaves it); with `out` (host) it waits for the device and copies the
 * last traced epoch: out[0] = GEMM tasks G, out[1] = stream tasks S, then per
 * task (the G GEMM tasks in their queue order, then the S stream tasks) six
 * words of %globaltimer ns: GEMM tasks -- dequeued, dependencies met, MMAs
 * started, last MMA issued, epilogue started, done; stream tasks --
 * dequeued, dependencies met, the SM that ran it (not a time), unused,
 * unused, done.  Returns the words written, 0 if there is no trace, -1 on an
 * error. */
FF_API long long ff_net_epoch_trace(ff_net* net, int enable, unsigned long long* out, long long capacity);

/* Makes `stream` wait for all work the net has enqueued so far.  The steps
 * enqueued between two ff_net_sync calls on one stream depend on nothing
 * outside them but that stream, so such a sequence can be captured into a
 * CUDA graph (the layers' workspaces must already be large enough). */
FF_API ff_status ff_net_sync(ff_net* net, void* stream);

/* Host-side bounded wait: blocks the calling thread until everything the net
 * has enqueued so far has finished (FF_OK) or timeout_ms milliseconds have
 * passed (FF_ERR_TIMEOUT; the work keeps running and a later wait can finish
 * it).  Polls event completion; takes no GPU-side wait of its own. */
FF_API ff_status ff_net_wait(ff_net* net, unsigned int timeout_ms);

/* ---------------------------------------------------------------------------
 * Allocation-free forward pass.  The paper has no counterpart: this is a
 * service for callers that cannot call cudaMalloc -- code embedded in a host
 * application that owns all device memory through its own pool, or that must
 * keep the device's memory footprint fixed after start-up -- and therefore
 * cannot create an ff_layer (which allocates its parameters and workspace).
 *
 * Computes what ff_layer_forward computes in FF_BF16 mode, from caller
 * buffers only: x [rows, ff_row_stride(in_features)] bf16 (16-byte aligned),
 * row_scale [rows] (required), W_bf16 [out_features, ff_row_stride(in_features)]
 * bf16, bias [out_features] fp32 or NULL, h_out [rows, ff_row_stride(out_features)]
 * bf16, goodness and next_scale [rows] or NULL, device_status [1] int or NULL
 * (set to 0 by the call, then OR-ed with 1 if a kernel wait timed out, 2 if a
 * goodness was not finite).  It allocates nothing: the per-tile goodness
 * partials live in a fixed 4 MiB array in the library's device image, which
 * every GPU that loads libff holds until the process exits.
 *   - Limit: rows * 2 * ceil(out_features / 256) <= 1048512 (two goodness
 *     partials per 256-column tile and row); larger requests return
 *     FF_ERR_INVALID_ARG before anything is enqueued.
 *   - Every call looks up that array's device address on the caller's
 *     current device (the lookup enqueues nothing).  The first call on a
 *     device also loads the library's device code there: make it before any
 *     stream capture.
 *   - rows == 0 computes nothing and still sets device_status to 0.
 *   - Every call shares the array and it keeps the last call's contents:
 *     calls whose work overlaps on the GPU (other streams, other threads)
 *     race; order them on one stream.
 *   - Needs an sm_100-family GPU (FF_ERR_UNSUPPORTED otherwise). */
FF_API ff_status ff_forward_noalloc(const void* x, const float* row_scale, const void* W_bf16,
                                    const float* bias, int rows, int in_features, int out_features,
                                    void* h_out, float* goodness, float* next_scale,
                                    int* device_status, void* stream);

/* Self-test of failure detection (the paper has no counterpart): enqueues on
 * `stream` one kernel that waits, through the same bounded mbarrier wait the
 * GEMM kernels use, on a barrier nothing arrives on.  After timeout_us
 * (1 .. 10 000 000) the wait gives up and latches the timeout in the layer;
 * ff_layer_check then returns FF_ERR_TIMEOUT and the context stays usable. */
FF_API ff_status ff_layer_selftest_wait(ff_layer* layer, unsigned int timeout_us, void* stream);

/* ---------------------------------------------------------------------------
 * Instrumentation (not part of the method).
 * Every kernel launch libff makes is counted; ff_kernel_launches returns the
 * process-wide total so far.  ff_profile_enable(1) clears earlier records and
 * starts bracketing each launch with two CUDA events recorded on the stream
 * the kernel is launched on; ff_profile_enable(0) stops.  ff_profile_read
 * waits for the recorded events and writes, for up to `capacity` kernel kinds
 * that were launched, the kind's name (static string), launch count, summed
 * device time in ms and summed algorithmic work (FLOPs for kinds whose name
 * contains "gemm", bytes the algorithm must move for the others).  Returns the
 * number of kinds written, or -1 if an event query failed.  Any output array
 * may be NULL. */
FF_API ff_status ff_profile_enable(int on);
FF_API int ff_profile_read(int capacity, const char** names, long long* launches, double* ms,
                           double* work);
FF_API unsigned long long ff_kernel_launches(void);
/* The recorded launches in order: kind id (ff_profile_kind_name gives its
 * name), launching stream (as an integer), start and end in ms relative to the
 * earliest recorded start.  Returns how many were written, or -1. */
FF_API int ff_profile_timeline(int capacity, int* kind, long long* stream_id, double* start_ms,
                               double* end_ms);
FF_API const char* ff_profile_kind_name(int kind);

#ifdef __cplusplus
}
#endif
#endif /* FF_H */
