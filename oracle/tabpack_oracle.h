/*
 * tabpack_oracle.h -- CPU fp64 oracle of one TabPack training step.
 *
 * TEST INFRASTRUCTURE ONLY.  This library is the slow, plain, obviously
 * correct restatement of the packed-ensemble method that the GPU library is
 * checked against.  Only the test suite, the smoke check and the benchmark's
 * CPU-baseline leg may load it; the product path never does.  It shares no
 * code, header, table or constant with the CUDA library.
 *
 * What it computes (paper: "TabPack: Efficient Hyperparameter Ensembles for
 * Tabular Deep Learning"):
 *   - a pack of m base MLPs, each a stack of Linear-ReLU-Dropout blocks with
 *     its own depth, width and dropout rate, followed by a linear head
 *     (Sec. 3.3 "Model Pack", Fig. 4 and Fig. 5 left);
 *   - per-member losses that are summed, never the predictions (Sec. 3.6
 *     "Training"): cross-entropy for classification, MSE for regression
 *     (Appendix F.1 "Experiment Setup");
 *   - exact backward pass (chain rule) and a pack of AdamW optimizers with
 *     per-member learning rate and weight decay (Sec. 3.4 "Optimizer Pack");
 *   - per-member validation predictions and greedy ensemble selection
 *     (Sec. 3.5 "Ensemble", "Greedy ensembling").
 *
 * All arithmetic is IEEE fp64 except where a mode says otherwise:
 *   - bf16_storage = 1 models the GPU's bf16 mode: the values the GPU stores
 *     in bf16 between kernels (the gathered batch, the weight copies fed to
 *     matrix products, hidden activations and back-propagated pre-activation
 *     gradients) are rounded to fp32 and then to bf16 (round to nearest even
 *     at both steps, as the GPU stores fp32 results in bf16) at the same
 *     points; every operation is still fp64.
 *   - orc_greedy(..., fp32_terms = 1) takes each per-row score term in fp32,
 *     the precision in which the GPU scorer takes the same decision.
 *
 * Parity status: every function here is pinned by tests in tests/ against
 * closed forms, finite differences, torch CPU fp64 library routines, brute
 * force or published values; Philox4x32-10 word by word by the known-answer
 * vectors published with Random123 (Salmon et al., SC'11), and structurally
 * (Weyl key constants from their closed forms, round invertibility).
 */
#ifndef TABPACK_ORACLE_H
#define TABPACK_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum { ORC_BINARY = 0, ORC_MULTICLASS = 1, ORC_REGRESSION = 2 };
enum { ORC_SCORE_LOSS = 0, ORC_SCORE_ACCURACY = 1, ORC_SCORE_RMSE = 2, ORC_SCORE_AUC = 3 };

/* ROC-AUC of scores e [N] (probability of class 1) for labels y [N] (0 / 1):
 * the scores are rounded to fp32 (the decision precision of the GPU scorer)
 * and ranked, tied scores sharing the mean of their ranks; AUC = (sum of the
 * positives' ranks - n_pos (n_pos + 1) / 2) / (n_pos n_neg) (Mann-Whitney).
 * NaN when one class is absent.  As an ensemble score (ORC_SCORE_AUC,
 * binary tasks) the greedy selection minimises -AUC.                        */
double orc_auc(const double* e, const int32_t* y, int64_t N);

typedef struct {
  int32_t m;            /* number of base models in the pack (the paper's m) */
  int32_t d_in;         /* input features */
  int32_t d_out;        /* 1 (binary, regression) or number of classes      */
  int32_t task;         /* ORC_BINARY / ORC_MULTICLASS / ORC_REGRESSION      */
  uint64_t seed;        /* Philox key for init and dropout                  */
  double beta1, beta2, eps;
  int32_t wd_on_bias;   /* 1: weight decay also applies to biases           */
  int32_t bf16_storage; /* 1: model the bf16 storage points of bf16 mode    */
} orc_config;

typedef struct orc_pack orc_pack;

/* Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11). */
void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]);

/* Dropout decision for element (row, col) of hidden layer `layer` (0-based)
 * of the member with stream id `member_id` at step `step`: 1 = keep.          */
int orc_dropout_keep(uint64_t seed, uint32_t member_id, uint32_t layer, uint32_t step,
                     uint32_t row, uint32_t col, float p);

/* orc_dropout_keep for rows 0..B-1, columns 0..w-1: out [B, w] uint8.   */
void orc_dropout_mask(uint64_t seed, uint32_t member_id, uint32_t layer, uint32_t step,
                      int32_t B, int32_t w, float p, uint8_t* out);

/* Round-to-nearest-even to bfloat16, result returned as a double. */
double orc_round_bf16(double x);

/* depth/width/dropout/lr/wd: length m host arrays, copied.  member_id: the
 * Philox stream id of each member (NULL: 0..m-1).  Parameters are initialised
 * from Philox (see orc_init_value).  Returns NULL on invalid arguments.       */
orc_pack* orc_create(const orc_config* cfg, const int32_t* depth, const int32_t* width,
                     const float* dropout, const float* lr, const float* wd,
                     const int32_t* member_id);
void orc_destroy(orc_pack* h);

/* The same pack with periodic feature embeddings (App. "Feature Embeddings"):
 * member i (d_emb[i] >= 1) maps feature j to alpha_j * [x_j, cos(w_j x_j +
 * b_j)] + beta_j in R^d_emb (w_j, b_j in R^(d_emb - 1); alpha_j, beta_j in
 * R^d_emb), and its first layer reads the d_in embeddings side by side
 * (d_in d_emb inputs, initialised like any layer of that fan-in).  freq: the
 * initial w of every member in turn, d_in x (d_emb[i] - 1) values each (the
 * caller draws them from N(0, sigma_i^2)); b, alpha, beta start at zero.
 * The embedding parameters take AdamW steps like biases.                     */
orc_pack* orc_create_emb(const orc_config* cfg, const int32_t* depth, const int32_t* width,
                         const float* dropout, const float* lr, const float* wd,
                         const int32_t* member_id, const int32_t* d_emb, const double* freq);
/* A member's embedding parameters (grads 0) or their last gradients
 * (grads 1): [w, b, alpha, beta] as above, d_in (4 d_emb - 2) values.        */
int orc_get_emb(const orc_pack* h, int32_t member, int32_t grads, double* out);
int orc_set_emb(orc_pack* h, int32_t member, const double* in);

/* Initial value of element e of layer `layer` (0-based; layer == depth is the
 * head) of a member, as stored (fp32-representable).                          */
double orc_init_value(uint64_t seed, uint32_t member_id, uint32_t layer, uint32_t e, int32_t fan_in);

/* One step: gather rows idx[0..B) of X [N, d_in] (fp32, row-major) and labels
 * (y_int for classification, y_float for regression; indexed like X), run the
 * forward, loss, backward and (if update) AdamW for every active member.
 * loss_out[i] (may be NULL) gets member i's mean loss (NaN if inactive).       */
int orc_train_step(orc_pack* h, const float* X, int64_t N, const int32_t* idx,
                   const int32_t* y_int, const float* y_float, int32_t B,
                   uint32_t step, int32_t update, double* loss_out);

/* The same step with a batch per member (Sec. 3.6: the base models train on
 * different batch sequences, one training batch being m base batches of B
 * rows stacked along the pack dimension): idx is [m, B], member i reads rows
 * idx[i * B .. i * B + B - 1] (rows of inactive members are still checked). */
int orc_train_step_stacked(orc_pack* h, const float* X, int64_t N, const int32_t* idx,
                           const int32_t* y_int, const float* y_float, int32_t B,
                           uint32_t step, int32_t update, double* loss_out);

/* Forward only, no dropout: out [m, N, d_out] = probabilities (softmax /
 * sigmoid) or regression values.                                               */
int orc_predict(orc_pack* h, const float* X, int64_t N, double* out);

int orc_set_active(orc_pack* h, const uint8_t* active);

/* Muon for the hidden-layer weight matrices (the paper's default optimizer,
 * Sec. 3.4 / App. F.1; AdamW stays on biases and the head): member i with
 * learning rate lr_muon[i], momentum mu (Nesterov), ns_steps Newton-Schulz
 * iterations; see tabpack_oracle.c for the steps.  Returns 0 on success.     */
int orc_set_muon(orc_pack* h, const double* lr_muon, double momentum, int32_t ns_steps);
/* The orthogonalized direction O of U [rows, cols] (bf16 != 0: rounding of
 * X, A and Bm to bf16 where the GPU stores them).                            */
void orc_newton_schulz(const double* U, int32_t rows, int32_t cols, int32_t steps, int32_t bf16, double* O);
/* The direction O [out, in] of the last Muon step of hidden layer `layer`.  */
int orc_get_muon_dir(const orc_pack* h, int32_t member, int32_t layer, double* out);

/* One AdamW step (PyTorch semantics, the update the training step applies to
 * every parameter; Sec. 3.4) on n elements in place: decoupled decay
 * p <- p - lr wd p, moments m, v, then the step bias-corrected for step
 * count t >= 1.                                                              */
void orc_adamw_apply(double* p, double* m, double* v, const double* g, int64_t n, int64_t t, double lr,
                     double wd, double beta1, double beta2, double eps);

/* layer in [0, depth] (depth = head).  W row-major [out, in], b [out].       */
int orc_get_params(const orc_pack* h, int32_t member, int32_t layer, double* W, double* b);
int orc_set_params(orc_pack* h, int32_t member, int32_t layer, const double* W, const double* b);
int orc_get_grads(const orc_pack* h, int32_t member, int32_t layer, double* W, double* b);
int orc_get_adam_state(const orc_pack* h, int32_t member, int32_t layer,
                       double* mW, double* vW, double* mb, double* vb);
/* logits of the last forward [B, d_out] */
int orc_get_logits(const orc_pack* h, int32_t member, double* out);
/* dropout keep mask of the last step for hidden layer `layer` [B, width] */
int orc_get_keep(const orc_pack* h, int32_t member, int32_t layer, uint8_t* out);
/* pre-activations Z of the last forward for hidden layer `layer` [B, width]   */
int orc_get_preact(const orc_pack* h, int32_t member, int32_t layer, double* out);
/* smallest |Z| / rms(Z) over the pre-activations of the last forward          */
double orc_get_margin(const orc_pack* h, int32_t member);
int64_t orc_member_steps(const orc_pack* h, int32_t member);

/* Greedy ensemble selection (Sec. 3.5).  preds [P, N, d_out] fp32.  Writes
 * the selection order to selected[0..*n_selected) and the final score.
 * step_best / step_gap (may be NULL, length m_ens): best score of each
 * iteration and its margin to the runner-up (+inf if there is none).          */
int orc_greedy(const float* preds, int32_t P, int64_t N, int32_t d_out,
               const int32_t* y_int, const float* y_float, int32_t task, int32_t score,
               int32_t m_ens, int32_t fp32_terms,
               int32_t* selected, int32_t* n_selected, double* final_score,
               double* step_best, double* step_gap);

/* Score of one fixed subset (plain definition, fp64). */
double orc_ensemble_score(const float* preds, const int32_t* subset, int32_t n_subset,
                          int64_t N, int32_t d_out, const int32_t* y_int, const float* y_float,
                          int32_t task, int32_t score);

#ifdef __cplusplus
}
#endif
#endif
