/*
 * tabpack.h -- C ABI of the GB300 (sm_103a) library for training a packed
 * hyperparameter ensemble of tabular MLPs, after "TabPack: Efficient
 * Hyperparameter Ensembles for Tabular Deep Learning".
 *
 * A pack holds m base MLPs ("base models", Sec. 3.3).  Member i is a stack of
 * depth[i] Linear-ReLU-Dropout blocks of width width[i] with dropout rate
 * dropout[i], followed by a linear head with d_out outputs; it is trained by
 * its own AdamW optimizer with learning rate lr[i] and weight decay wd[i]
 * (the optimizer pack, Sec. 3.4).  All members see the same input batch and
 * are trained independently: the per-member losses are summed, so each
 * member's gradient is that of its own loss (Sec. 3.6 "Training").
 *
 * Conventions for every entry point:
 *   - Pointers documented "device" are CUDA device pointers; they are read or
 *     written asynchronously on the pack's stream and must stay valid until
 *     the work on that stream has finished.  Pointers documented "host" are
 *     ordinary host memory, read or written before the call returns.
 *   - The caller owns every pointer argument; the pack owns its own device
 *     memory (parameters, optimizer state, activations), allocated at
 *     pack_create and freed at pack_destroy.
 *   - Matrices are row-major.  Weights of a layer are [out, in]; biases [out].
 *     Layer index l is 0-based: 0 .. depth-1 are the hidden blocks and
 *     l == depth is the head.
 *   - Labels y are device int32 class indices (binary: 0/1, multiclass:
 *     0..d_out-1) or device float32 targets (regression), with one entry per
 *     row of X.
 *   - No C++ exception crosses the ABI.  Every entry point returns a
 *     tp_status; on failure pack_last_error() describes the cause.  A
 *     TP_ECUDA status means a CUDA call failed; the pack should then be
 *     destroyed.
 *   - A pack is not thread-safe: use it from one host thread at a time.
 */
#ifndef TABPACK_H
#define TABPACK_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct tabpack tabpack_t;

typedef enum {
  TP_OK = 0,
  TP_EINVAL = 1,    /* an argument is out of range or inconsistent        */
  TP_ENOMEM = 2,    /* device or pinned-host allocation failed            */
  TP_ECUDA = 3,     /* a CUDA runtime/driver call failed                  */
  TP_ESTATE = 4,    /* call not valid in the pack's current state         */
  TP_ETIMEOUT = 5,  /* a bounded device-side wait gave up                 */
  TP_ENOTSUP = 6    /* configuration not supported on this device         */
} tp_status;

typedef enum { TP_BINARY = 0, TP_MULTICLASS = 1, TP_REGRESSION = 2 } tp_task;
typedef enum { TP_BF16 = 0, TP_FP32 = 1 } tp_precision;
typedef enum { TP_SCORE_LOSS = 0, TP_SCORE_ACCURACY = 1, TP_SCORE_RMSE = 2, TP_SCORE_AUC = 3 } tp_score;

typedef struct {
  int32_t m;          /* number of base models in the pack, >= 1                        */
  int32_t d_in;       /* input features, >= 1                                           */
  int32_t d_out;      /* 1 for binary / regression, number of classes (2..32) otherwise  */
  int32_t max_batch;  /* largest B passed to pack_train_step, >= 1                      */
  int32_t task;       /* tp_task                                                        */
  int32_t precision;  /* tp_precision: TP_BF16 runs the matrix products on bf16 tensor
                         cores with fp32 accumulation and stores activations in bf16;
                         TP_FP32 keeps everything in fp32 (CUDA-core products)           */
  uint64_t seed;      /* Philox key of parameter init and dropout masks                 */
  float beta1, beta2, eps;  /* AdamW constants shared by all members (0.9, 0.999, 1e-8) */
  int32_t wd_on_bias; /* 1: weight decay also applies to biases                         */
  int32_t fuse_optimizer; /* bf16 mode only.  0: the weight-gradient products store fp32
                         gradients and one AdamW pass updates all parameters (faster on
                         most shapes); 1: AdamW runs inside the weight-gradient product's
                         epilogue, so gradients never reach HBM.  Results are the same. */
} tp_config;

/* Create a pack (Sec. 3.3 model pack + Sec. 3.4 optimizer pack).
 * depth, width, dropout, lr, wd: host arrays of length cfg->m, copied.
 *   depth[i] in 1..14; width[i] a positive multiple of 16 (<= 4096);
 *   0 <= dropout[i] < 1; lr[i] >= 0; wd[i] >= 0.
 * cuda_stream: the cudaStream_t all work of this pack runs on (NULL: the
 *   legacy default stream).
 * Parameters are initialised on the device from Philox4x32-10: element e of
 * layer l of member i (weights row-major, then biases) takes the word at
 * counter (e >> 2, 0, 0, 1 << 28 | i << 4 | l), word e & 3, key cfg->seed;
 * with u = ((r >> 8) + 1/2) 2^-24 its value is (2u - 1) / sqrt(fan_in),
 * rounded to fp32 (U(-1/sqrt(fan_in), 1/sqrt(fan_in)), the PyTorch Linear
 * default; the paper does not state its init).
 * On success *out receives the handle; on failure *out is NULL.             */
tp_status pack_create(const tp_config* cfg, const int32_t* depth, const int32_t* width,
                      const float* dropout, const float* lr, const float* wd,
                      void* cuda_stream, tabpack_t** out);

/* Create a pack whose members read periodic feature embeddings (App.
 * "Feature Embeddings"): feature j of member i becomes the d = d_emb[i]
 * values  alpha_j (.) [x_j, cos(w_j x_j + b_j)] + beta_j  (w_j, b_j of
 * length d - 1; alpha_j, beta_j of length d; (.) elementwise), and the
 * first hidden layer reads the d_in embeddings side by side (column j d + k
 * is component k of feature j), so its input width is d_in d.
 * Arguments as pack_create, plus d_emb: host [m], each in 1..64; freq: host
 * array holding, member after member, the d_in (d_emb[i] - 1) initial
 * frequencies w of member i (row-major [d_in, d_emb[i] - 1]; the paper
 * draws them from N(0, sigma), sigma a per-member hyperparameter, so the
 * caller draws them); b, alpha and beta start at zero.  The embedding
 * parameters are trained by AdamW with the member's lr, as the biases are
 * (weight decay on them only when cfg->wd_on_bias), also under Muon;
 * fuse_optimizer is turned off.  The embedding kernels compute in fp32
 * (cosf) and store E in the matrix-product precision; their gradients
 * are accumulated in fp64 over the batch rows in order.  Memory: an
 * embedding matrix [max_batch rounded up to 128, d_in d rounded up to 8,
 * plus 16] per member, its input gradient, and, while predicting, the
 * same for a chunk of at most 8192 rows, fewer where the chunk's
 * embedding matrices of all members would pass 1 GiB.                    */
tp_status pack_create_emb(const tp_config* cfg, const int32_t* depth, const int32_t* width,
                          const float* dropout, const float* lr, const float* wd, const int32_t* d_emb,
                          const float* freq, void* cuda_stream, tabpack_t** out);

/* Member `member`'s embedding parameters (grads = 1: their gradients from
 * the last step; a pack with embeddings stores them on every step, since
 * its optimizer runs as a separate pass), copied to the host array out of
 * d_in (4 d - 2) floats: w [d_in, d - 1], b [d_in, d - 1], alpha [d_in, d],
 * beta [d_in, d], d = its d_emb.  TP_EINVAL for a pack without
 * embeddings.  Synchronises.                                                */
tp_status pack_get_emb(tabpack_t* pack, int32_t member, int32_t grads, float* out);
/* Overwrite member `member`'s embedding parameters from the host array in
 * (layout of pack_get_emb).  Synchronises.                                 */
tp_status pack_set_emb(tabpack_t* pack, int32_t member, const float* in);
/* *d_emb = member `member`'s embedding size (0 for a pack without). */
tp_status pack_member_emb(const tabpack_t* pack, int32_t member, int32_t* d_emb);

/* Free the pack and its device memory (waits for the pack's stream). NULL ok. */
void pack_destroy(tabpack_t* pack);

/* Change the stream subsequent work is enqueued on. */
tp_status pack_set_stream(tabpack_t* pack, void* cuda_stream);

/* One training step of every active member (Sec. 3.6): gather rows
 * idx[0..B) of X, forward through each member's blocks with its own dropout
 * rate, per-member mean loss (cross-entropy for multiclass, logistic loss on
 * one logit for binary, MSE for regression), backward, and one AdamW update
 * per member with its own lr and wd and its own step count t (PyTorch AdamW
 * semantics: p <- p - lr wd p, then the bias-corrected Adam step).
 *   X: device float32 [n_rows, d_in];  idx: device int32 [B], 0 <= idx < n_rows
 *   (not checked on the device);  y: device labels [n_rows] (see above);
 *   1 <= B <= max_batch;  step: dropout counter of this step (masks are a
 *   function of (seed, member, layer, step, row, col): keep iff the Philox
 *   word at counter (row, col >> 2, step, member << 4 | layer), word col & 3,
 *   is >= floor(dropout * 2^32));
 *   loss_out: device float32 [m] (may be NULL): member i's mean loss, NaN for
 *   inactive members.
 * Asynchronous: returns once the work is enqueued.                          */
tp_status pack_train_step(tabpack_t* pack, const float* X, int64_t n_rows, const int32_t* idx,
                          const void* y, int32_t B, uint32_t step, float* loss_out);

/* Same as pack_train_step without the optimizer update: the gradients of
 * the step stay readable through pack_get_grads and the step counts do not
 * advance.  For tests and diagnostics.                                       */
tp_status pack_forward_backward(tabpack_t* pack, const float* X, int64_t n_rows, const int32_t* idx,
                                const void* y, int32_t B, uint32_t step, float* loss_out);

/* The same steps with a batch per member (Sec. 3.6: the base models are
 * trained on different batch sequences; one training batch is m base
 * batches of B rows stacked along the pack dimension).
 *   idx: device int32 [m, B]: member i's batch is rows idx[i * B .. i * B +
 *   B - 1] of X (rows of inactive members are not read; no range check on
 *   the device).  Everything else as pack_train_step / pack_forward_backward;
 *   dropout masks are the same function of (seed, member, layer, step, row
 *   position, column).  The first call allocates m gathered-batch matrices
 *   ([max_batch rounded up to 128, d_in rounded up to 8, plus 16] each, in
 *   the matrix-product precision) and synchronises.                         */
tp_status pack_train_step_stacked(tabpack_t* pack, const float* X, int64_t n_rows, const int32_t* idx,
                                  const void* y, int32_t B, uint32_t step, float* loss_out);
tp_status pack_forward_backward_stacked(tabpack_t* pack, const float* X, int64_t n_rows, const int32_t* idx,
                                        const void* y, int32_t B, uint32_t step, float* loss_out);

/* Muon for the hidden-layer weight matrices (the paper's default optimizer:
 * Muon for the weights of the hidden linear layers, AdamW for biases and the
 * head; Sec. 3.4, App. F.1; Jordan et al. 2024), from the next step on.
 * Per step and matrix W [out, in] with gradient G:
 *   M <- mu M + (1 - mu) G;  U = (1 - mu) G + mu M (Nesterov);
 *   X = U / max(||U||_F, 1e-7), transposed when out > in;
 *   ns_steps times: A = X X^T; Bm = b A + c A A; X = a X + Bm X,
 *   (a, b, c) = (3.4445, -4.7750, 2.0315) (on the tensor cores in bf16 mode,
 *   X, A and Bm stored in bf16, and U stored as X with 1 / max(||U||_F,
 *   1e-7) applied in fp32 inside the first iteration's products; on CUDA
 *   cores in fp32 mode);
 *   W <- W - lr_muon wd W;  W <- W - lr_muon max(1, out / in)^(1/2) X
 * (in = the real input width).  lr_muon: host [m]; wd: the member's weight
 * decay; momentum in [0, 1); ns_steps in 1..32 (5 in the paper's Muon).  The
 * momentum buffers start at zero; AdamW in the weight-gradient epilogue
 * (fuse_optimizer) is turned off.  Allocates the Newton-Schulz buffers
 * (2 r c + 2 r^2 elements per matrix, r = min(out, in), c = max) on the
 * first call; synchronises.  TP_EINVAL when a matrix has 2^31 elements or
 * more (out times the input width rounded up to 8).                         */
tp_status pack_set_muon(tabpack_t* pack, const float* lr_muon, float momentum, int32_t ns_steps);

/* The direction X of the last Muon step of hidden layer `layer` of `member`
 * (the orthogonalised momentum, [out, in] with the real input width):
 * host float32.  For tests and diagnostics; synchronises.                    */
tp_status pack_debug_muon_dir(tabpack_t* pack, int32_t member, int32_t layer, float* out);

/* Per-member validation predictions (Sec. 3.5 "Online ensemble"): forward
 * without dropout of every active member on all N rows of X.
 *   X: device float32 [N, d_in];  out: device float32 [m, N, d_out]:
 *   softmax probabilities (multiclass), sigmoid probability of class 1
 *   (binary) or the regression value.  Rows of inactive members are left
 *   untouched.  Asynchronous.                                                */
tp_status pack_predict(tabpack_t* pack, const float* X, int64_t N, float* out);

/* Greedy ensemble selection over a pool of P candidates (Sec. 3.5 "Greedy
 * ensembling"): start from the candidate with the best ensemble score, then
 * repeatedly add the unused candidate whose addition gives the best score of
 * the averaged prediction; stop after m_ens members or when the best
 * addition does not strictly improve the score.  Ties go to the lowest
 * candidate index.  Scores (lower is better): TP_SCORE_LOSS = mean CE / BCE
 * of the averaged probabilities clipped to [1e-7, 1 - 1e-7], or MSE;
 * TP_SCORE_ACCURACY = minus the accuracy (classification);
 * TP_SCORE_RMSE = root MSE (regression); TP_SCORE_AUC = minus the ROC-AUC
 * (binary): the ensemble's scores rounded to fp32 are ranked (stable radix
 * sort on the device), tied scores share their mean rank, and AUC = (sum of
 * the positives' ranks - n_pos (n_pos + 1) / 2) / (n_pos n_neg) (NaN, never
 * selected, when a class is absent).  Per-row terms are taken in fp32 and
 * summed in fp64 in a fixed order; the running ensemble sum is fp64.
 *   preds: device float32 [P, N, d_out] (probabilities or values as written
 *   by pack_predict);  y: device labels [N];  cuda_stream: stream to run on;
 *   selected: host int32 [m_ens] receives the selection order;
 *   n_selected, final_score: host outputs.
 * Allocates its scratch with cudaMallocAsync on the stream and synchronises
 * the stream before returning.                                              */
tp_status pack_select_greedy(const float* preds, int32_t P, int64_t N, int32_t d_out, const void* y,
                             int32_t task, int32_t score, int32_t m_ens, void* cuda_stream,
                             int32_t* selected, int32_t* n_selected, double* final_score);

/* pack_select_greedy without any memory allocation.  (The paper has no
 * counterpart: this is a deployment variant of the same selection.)
 * Same arguments, results and stream behaviour as pack_select_greedy, but
 * the scratch lives in one fixed 16 MiB array of device memory that the
 * library defines at file scope; every GPU that loads the library holds it
 * until the process exits.  It is for callers that cannot call cudaMalloc /
 * cudaMallocAsync when they select: processes whose device memory is already
 * fully reserved by another framework's caching allocator, loops that must
 * not risk an out-of-memory failure or an allocator synchronisation, and
 * embedding runtimes that forbid allocation calls after start-up.  It calls
 * no allocating routine.
 *   Limit: the problem must fit, N*d_out*8 + P*ceil(N/1024)*8 +
 *   (4 + m_ens + P)*4 + 1024 <= 16 MiB, with P*N*10 + 512 more bytes for
 *   TP_SCORE_AUC (its sort keys and labels); e.g. N = 100000 rows of 10
 *   classes with P = 96 candidates, or ROC-AUC on N = 20000 rows with P = 80.
 *   Larger problems return TP_EINVAL with the exact need in the message of
 *   pack_last_error(NULL) and do nothing.
 *   The first call on each device (and the first after a device reset)
 *   looks up the array's device address (cudaGetSymbolAddress, with that
 *   device current); make that first call before any stream capture.
 *   selected receives the *n_selected selected slots only.
 *   All calls share the one array and each call starts by clearing what it
 *   needs, so calls that overlap on the GPU (concurrent streams) race and
 *   must be serialised by the caller.                                        */
tp_status pack_select_greedy_static(const float* preds, int32_t P, int64_t N, int32_t d_out, const void* y,
                                    int32_t task, int32_t score, int32_t m_ens, void* cuda_stream,
                                    int32_t* selected, int32_t* n_selected, double* final_score);

/* Base-model early stopping hook (Sec. 3.6): active is a host uint8 [m];
 * inactive members are skipped by every kernel and keep their parameters,
 * optimizer state and step count.                                           */
tp_status pack_set_active(tabpack_t* pack, const uint8_t* active);

/* Copy one layer's fp32 master parameters to / from host memory.
 * W: host float32 [out, in] (may be NULL), b: host float32 [out] (may be
 * NULL).  Synchronises the pack's stream.  pack_set_params also refreshes
 * the bf16 copy used by the tensor-core products.                           */
tp_status pack_get_params(tabpack_t* pack, int32_t member, int32_t layer, float* W, float* b);
tp_status pack_set_params(tabpack_t* pack, int32_t member, int32_t layer, const float* W, const float* b);

/* Member snapshots (the "intermediate base-model checkpoints" of Sec. 3.5
 * that the online ensemble keeps).  Member i's fp32 master parameters are
 * one contiguous run of the pack's parameter arena, of *n_elems elements:
 * for l = 0 .. depth[i] in turn, the weights [out, in_pad] row-major and
 * then the bias [out], each block starting at a multiple of 32 elements
 * from the start of the run, the gaps zero; in_pad = d_in rounded up to a
 * multiple of 8 for l = 0 (pad columns zero), width[i] otherwise.  The run
 * depends only on (d_in, d_out, depth[i], width[i]), so a snapshot of one
 * pack restores into any member of the same shape in any pack.
 *   pack_snapshot: copies the run to dst, a device float32 buffer of
 *     *n_elems elements; asynchronous on the pack's stream (device to
 *     device), so it captures the state after all work enqueued before it.
 *   pack_restore: copies a run written by pack_snapshot back from src
 *     (device) and refreshes the bf16 weight copies; synchronises.  The
 *     member's optimizer state and step count are left as they are.      */
tp_status pack_member_size(const tabpack_t* pack, int32_t member, int64_t* n_elems);
tp_status pack_snapshot(tabpack_t* pack, int32_t member, float* dst);
tp_status pack_restore(tabpack_t* pack, int32_t member, const float* src);

/* Read back what pack_create was given: the configuration, one member's
 * hyperparameters (any output pointer may be NULL), the active mask (host
 * uint8 [m], 1 = trained) and the stream the pack runs on.                 */
tp_status pack_get_config(const tabpack_t* pack, tp_config* cfg);
tp_status pack_member_hparams(const tabpack_t* pack, int32_t member, int32_t* depth, int32_t* width,
                              float* dropout, float* lr, float* wd);
tp_status pack_get_active(const tabpack_t* pack, uint8_t* active);
void* pack_get_stream(const tabpack_t* pack);

/* Gradients of the last pack_forward_backward, same layout as the params.  */
tp_status pack_get_grads(tabpack_t* pack, int32_t member, int32_t layer, float* W, float* b);

/* Logits of the last step for one member: host float32 [B, d_out].        */
tp_status pack_get_logits(tabpack_t* pack, int32_t member, float* out);

/* Dropout keep mask (1 keep, 0 drop) that step `step` applies to hidden
 * layer `layer` of `member`, evaluated on the device by the same function
 * the forward epilogue uses: host uint8 [B, width].                        */
tp_status pack_debug_masks(tabpack_t* pack, int32_t member, int32_t layer, uint32_t step,
                           int32_t B, uint8_t* keep);

/* Activations of the last forward for hidden layer `layer` of `member`
 * (the stored output of that layer, after ReLU and dropout): host float32
 * [B, width] with B the last step's batch size.  For tests and diagnostics. */
tp_status pack_debug_activations(tabpack_t* pack, int32_t member, int32_t layer, float* out);

/* The dropout keep mask held in the pack's mask arena for hidden layer
 * `layer` of `member` (bf16 mode): the words the forward epilogue reads
 * (Sec. 3.3, one mask per member at its own rate), decoded to host uint8
 * keep [B, width] (1 keep, 0 drop) for rows 0 .. B-1 (B <= max_batch).
 * *step_held receives the step whose masks the arena holds (-1: none yet).
 * After a training step t the arena holds step t + 1's masks (the optimizer
 * pass fills them), which the forward of step t + 1 then reads unchanged;
 * after pack_forward_backward(t) it holds step t's, the ones that forward
 * applied.  Layers with rate 0 report all ones.  TP_ESTATE in fp32 mode,
 * whose epilogue evaluates the keep bits itself.  Synchronises.            */
tp_status pack_debug_mask_arena(tabpack_t* pack, int32_t member, int32_t layer, int32_t B, uint8_t* keep,
                                int64_t* step_held);

/* Failure detection of the tensor-core products, for tests (the paper has
 * no counterpart).  Every wait of the persistent GEMM launches that can give
 * up gives up after wait_s seconds (default 2) -- the producer's waits for a
 * free stage or a row-block dependency -- or 2 wait_s -- the MMA and
 * epilogue waits, which wait on the producer: the CTA raises its abort flag, records the
 * wait's site code in the pack's device error word, lets its own copies and
 * MMAs finish, frees its tensor memory and exits, and the next
 * synchronising call returns TP_ETIMEOUT naming the site (3: a row-block
 * dependency).  poison != 0 also makes the first forward tile that waits
 * on a dependency wait for a count the launch never reaches, so the next
 * bf16 step's forward launch gives up there; the pack's results are then
 * undefined and it should be destroyed.  bf16 mode; synchronises; captured
 * step graphs are dropped.                                                 */
tp_status pack_debug_gemm_timeout(tabpack_t* pack, double wait_s, int32_t poison);

/* Where the bf16 tensor-core weight-gradient products take each hidden
 * layer's bias gradient db_j = sum_b dZ[b, j] (Sec. 3.3 backward; the paper
 * has no counterpart for the choice).  mode 1: for every layer whose input
 * width is a multiple of 256, from column sums of dZ that the head kernel
 * and the dgrad epilogues store while they write dZ (this saves a column
 * tile of the product); mode 0: from a column of ones appended to the
 * product's input, for every layer; mode -1: the pack's own choice (column
 * sums when its backward products are tensor-bound: ideal tensor time of
 * 300 us or more per step).  Both sum dZ as stored in bf16, in fp32.  For
 * tests and measurements; bf16 mode only (TP_ESTATE otherwise), TP_EINVAL
 * for another mode.  Synchronises; captured step graphs are dropped.      */
tp_status pack_debug_bias_path(tabpack_t* pack, int32_t mode);

/* Philox4x32-10 (Salmon et al., SC'11) as the device evaluates it for the
 * dropout masks and the initial values: out[i] = the four words of counter
 * ctr[i] (host uint32 [n, 4]) under key key[i] (host uint32 [n, 2]).  Runs
 * on the current device's default stream and synchronises; for tests.     */
tp_status pack_debug_philox(const uint32_t* ctr, const uint32_t* key, int32_t n, uint32_t* out);

/* Per-kernel-family timing with CUDA events recorded on the pack's stream.
 * Enable, run work, then read the accumulated milliseconds and launch counts
 * (synchronises).  Families: see tp_phase.                                  */
typedef enum {
  TP_PH_GATHER = 0, TP_PH_FWD = 1, TP_PH_HEAD = 2, TP_PH_BWD = 3, TP_PH_BIAS = 4,
  TP_PH_ADAMW = 5, TP_PH_PREDICT = 6, TP_PH_MUON = 7, TP_PH_COUNT = 8
} tp_phase;
tp_status pack_profile_enable(tabpack_t* pack, int32_t enable);
tp_status pack_profile_read(tabpack_t* pack, double* ms /* [TP_PH_COUNT] */,
                            int64_t* launches /* [TP_PH_COUNT] */, int32_t reset);

/* Number of kernels this pack has launched since creation.                 */
int64_t pack_launch_count(const tabpack_t* pack);

/* Sizes of the pack: number of fp32 parameters (as stored, including the
 * zero padding of layer-0 columns to a multiple of 8) and device bytes held. */
tp_status pack_sizes(const tabpack_t* pack, int64_t* n_params, int64_t* device_bytes);

/* ------------------------------------------------------------------------
 * Online ensemble (Sec. 3.5 "Online ensemble", Sec. 3.6 early stopping).
 *
 * The caller trains the pack for one epoch (pack_train_step over its
 * batches) and then calls pack_online_epoch, which
 *   1. predicts every active member on the validation rows (pack_predict);
 *   2. forms the candidate pool: the active members' current states
 *      (candidates 0 .. m-1, inactive members excluded) followed by the
 *      previous epoch's ensemble members in their selection order
 *      (candidates m, m+1, ...; their predictions are kept from the epoch
 *      they were made in), each an instance (member, epoch);
 *   3. rebuilds the ensemble from scratch by greedy selection over the pool
 *      (pack_select_greedy's rule and arithmetic, at most m_ens members);
 *      instances of the same member from different epochs are distinct
 *      candidates;
 *   4. snapshots the parameters of every newly selected current state
 *      (pack_snapshot into memory the object owns);
 *   5. base-model early stopping: a member's validation score is the score
 *      of its own prediction alone (the same score function); a score that
 *      is strictly below the member's best so far resets its count of
 *      non-improving epochs, any other (including NaN) increments it, and a
 *      member whose count reaches p_base + 1 is made inactive
 *      (pack_set_active) after this epoch's selection;
 *   6. ensemble early stopping: the same rule on the ensemble's score with
 *      p_ens; the best ensemble so far (lowest score, earliest on ties) is
 *      kept with its snapshots.  *stop becomes 1 when the count reaches
 *      p_ens + 1 or no member remains active.
 * Epochs are numbered from 1.  Scores are lower-is-better as in
 * pack_select_greedy.  The object works on the pack's stream; the pack must
 * outlive it.  Device memory it holds: the pool (m + 2 m_ens) * n_val *
 * d_out floats, 2 m_ens snapshot slots of the largest member's run, and
 * its selection scratch.                                                    */
typedef struct tabpack_online tabpack_online_t;

typedef struct {
  int32_t epoch;        /* epochs processed                                     */
  int32_t stop;         /* 1 once training should stop (see above)              */
  int32_t n_active;     /* members still trained                                */
  int32_t ens_bad;      /* consecutive epochs without ensemble improvement      */
  int32_t best_epoch;   /* epoch whose ensemble is the best (0: none yet)       */
  int32_t n_best;       /* members of the best ensemble                         */
  int32_t n_last;       /* members of the last epoch's ensemble                 */
  int32_t n_pool;       /* candidates in the last epoch's pool                  */
  double best_score;    /* score of the best ensemble (+inf: none yet)          */
  double last_score;    /* score of the last epoch's ensemble                   */
} tp_online_info;

/* Create the online ensemble of `pack` for validation sets of n_val rows.
 * score: tp_score (as pack_select_greedy; valid for the pack's task);
 * m_ens >= 1; p_base, p_ens >= 0 (the paper's defaults are 16 and 32).     */
tp_status pack_online_create(tabpack_t* pack, int64_t n_val, int32_t score, int32_t m_ens, int32_t p_base,
                             int32_t p_ens, tabpack_online_t** out);
void pack_online_destroy(tabpack_online_t* online);

/* End of an epoch (steps 1-6 above).  X_val: device float32 [n_val, d_in];
 * y_val: device labels [n_val]; stop: host output (may be NULL).
 * Synchronises the pack's stream.  After *stop = 1 further calls return
 * TP_ESTATE.                                                               */
tp_status pack_online_epoch(tabpack_online_t* online, const float* X_val, const void* y_val, int32_t* stop);

tp_status pack_online_info(const tabpack_online_t* online, tp_online_info* info);

/* Per-member state after the last epoch, host arrays of length m (any may be
 * NULL): score (the member's last validation score; NaN if it was inactive
 * in that epoch), best (its best score so far; +inf if none), bad (its count
 * of non-improving epochs).                                                */
tp_status pack_online_members(const tabpack_online_t* online, double* score, double* best, int32_t* bad);

/* An ensemble as instances: which = 0 the best ensemble, 1 the last
 * epoch's.  member, epoch: host int32 [m_ens] in selection order (may be
 * NULL); *n: its size; *score: its score (may be NULL).                     */
tp_status pack_online_ensemble(const tabpack_online_t* online, int32_t which, int32_t* member, int32_t* epoch,
                               int32_t* n, double* score);

/* Parameter run of instance j of the best ensemble (layout as
 * pack_snapshot; pack_member_size of its member gives the length) copied to
 * dst (device).  Synchronises.                                             */
tp_status pack_online_snapshot(tabpack_online_t* online, int32_t j, float* dst);

/* Prediction of the best ensemble on N rows: for every row the mean of its
 * n instances' predictions (probabilities or values as pack_predict writes
 * them), summed in fp64 in selection order and multiplied by 1/n, rounded
 * to fp32.  The instances run from their snapshots in a second pack the
 * object builds (and rebuilds when the best ensemble changes).
 *   X: device float32 [N, d_in];  out: device float32 [N, d_out].
 * Asynchronous on the pack's stream.                                       */
tp_status pack_online_predict(tabpack_online_t* online, const float* X, int64_t N, float* out);

/* Description of the last error of this online object.                    */
const char* pack_online_last_error(const tabpack_online_t* online);

/* Description of the last error on this pack (or, for pack == NULL, of the
 * last failed pack_create / pack_select_greedy / pack_select_greedy_static
 * on this thread).                                                         */
const char* pack_last_error(const tabpack_t* pack);

#ifdef __cplusplus
}
#endif
#endif
