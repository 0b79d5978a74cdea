/*
 * pnn.h -- C ABI of the GB300 parareal neural network training library.
 *
 * The library trains the parareal network f-bar of Lee, Lee & Park,
 * "Parareal Neural Networks Emulating a Parallel-in-time Algorithm"
 * (Section 3, eq:barf): a feed-forward CNN f = h o g o C is torn into N
 * consecutive subnetworks g^j (Section 3.1); all N run at once on one GPU
 * (Algorithm 1's parallel loop becomes grouped kernel launches), and the
 * coarse network F^j joins them through the parareal correction eq:correct.
 * The gradient follows Algorithm 2 (Section 3.2) and the update is SGD with
 * Nesterov momentum and weight decay (Section 4).
 *
 * Conventions shared by every call:
 *   - Every call returns a pnn_status; the library never aborts or exits.
 *     pnn_last_error() returns a human-readable message for the last failure.
 *   - Device pointers are CUDA device addresses of the current device; host
 *     pointers are ordinary (pageable or pinned) host memory.
 *   - All GPU work is enqueued on the stream given in pnn_options (NULL = the
 *     legacy default stream).  Calls marked "synchronises" wait for it.
 *   - The library owns the plan; the caller owns the workspace (one device
 *     allocation, see pnn_workspace_bytes / pnn_bind_workspace), which holds
 *     every parameter, gradient, momentum buffer, activation and table.
 *   - Tensors at the boundary are NCHW float32.  Inside, activations are NHWC.
 *   - A handle is not thread-safe.
 */
#ifndef PNN_H_
#define PNN_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct pnn_net pnn_net; /* opaque, library-owned */

typedef enum {
  PNN_OK = 0,
  PNN_EINVAL = 1,     /* bad argument or description */
  PNN_ENOMEM = 2,     /* workspace too small */
  PNN_ECUDA = 3,      /* a CUDA runtime call failed (message in pnn_last_error) */
  PNN_ESTATE = 4,     /* call out of order (e.g. backward before forward) */
  PNN_ETIMEOUT = 5,   /* a device-side bounded wait gave up */
  PNN_ENONFINITE = 6, /* loss is NaN/Inf or a label is out of range */
  PNN_ENOTBOUND = 7   /* no workspace bound yet */
} pnn_status;

typedef enum { PNN_BF16 = 0, PNN_FP32_CHECK = 1 } pnn_precision;

/* Section 3.1 eq:correct (default) or the classic parareal update of
 * Section 2 written for the residual: rt_{j+1} = r_{j+1} + F^j(x_{j+1}+rt_j) - F^j(x_{j+1}). */
typedef enum { PNN_CORR_RESIDUAL = 0, PNN_CORR_DELTA = 1 } pnn_correction;

/* Layer kinds of a description (Section 4, Tables vgg and resnet).  Every
 * conv is bias-free, k x k with zero padding k/2.
 *   PNN_CONV            bare conv (cout, k, stride)
 *   PNN_CONV_BN_RELU    conv -> BN -> ReLU, then a 2x2/s2 maxpool if pool != 0
 *   PNN_BASIC           post-activation basic block: ReLU(BN(conv(ReLU(BN(conv x)))) + x)
 *   PNN_BOTTLENECK      pre-activation bottleneck (cout, mid, stride on the 3x3
 *                       conv, 1x1 projection shortcut when the shape changes)
 *   PNN_COARSE_RU       coarse RU of Parareal ResNet (Section 4.2): two 3x3 convs
 *                       and a skip, in pre-activation order
 *                       conv3x3(ReLU(BN(conv3x3_s(ReLU(BN x))))) + skip, the
 *                       stride on the first conv, the skip a 1x1 (strided)
 *                       projection of ReLU(BN x) when the shape changes */
typedef enum {
  PNN_CONV = 0, PNN_CONV_BN_RELU = 1, PNN_BASIC = 2, PNN_BOTTLENECK = 3, PNN_COARSE_RU = 4
} pnn_layer_op;

/* Postprocessing h (eq:barf's epsilon part) */
typedef enum { PNN_HEAD_GAP_FC = 0, PNN_HEAD_BN_RELU_GAP_FC = 1, PNN_HEAD_GAP_MLP = 2 } pnn_head_kind;

/* What follows the 1x1 conv of C^j for j > 1 (Section 4.1 / 4.2: maxpools
 * 3x3/s2 down to the size of X_{j-1}, then a 1x1 conv). */
typedef enum { PNN_CJ_NONE = 0, PNN_CJ_BN_RELU = 1 } pnn_cj_post;

typedef struct {
  int32_t op;     /* pnn_layer_op */
  int32_t cout;   /* output channels */
  int32_t mid;    /* bottleneck width (PNN_BOTTLENECK only) */
  int32_t k;      /* kernel size (PNN_CONV, PNN_CONV_BN_RELU): 1 or 3 */
  int32_t stride; /* 1 or 2 */
  int32_t pool;   /* PNN_CONV_BN_RELU: non-zero appends a 2x2/s2 maxpool */
} pnn_layer;

/* A network description (Section 3.1):
 *   stem     the preprocessing operator C_delta = C^1
 *   body     the block-repetitive part g, torn into n_seg consecutive segments
 *            of segments[j] layers each (g^1 .. g^N)
 *   coarse   F^1 .. F^{N-1} concatenated; coarse_len[j] layers each
 *   head     h; head_hidden lists hidden FC widths for PNN_HEAD_GAP_MLP.
 * Arrays are read during pnn_create only. */
typedef struct {
  int32_t batch, in_c, in_h, in_w, classes;
  const pnn_layer* stem;
  int32_t n_stem;
  const pnn_layer* body;
  int32_t n_body;
  const int32_t* segments;
  int32_t n_seg;
  const pnn_layer* coarse;
  const int32_t* coarse_len; /* n_seg - 1 entries */
  int32_t cj_post;           /* pnn_cj_post */
  int32_t head_kind;         /* pnn_head_kind */
  const int32_t* head_hidden;
  int32_t n_hidden;
} pnn_desc;

typedef struct {
  int32_t precision;     /* pnn_precision */
  int32_t correction;    /* pnn_correction */
  uint64_t seed;         /* He-normal initialisation seed */
  float lr, momentum, weight_decay;
  int32_t nesterov;
  int32_t stream_fp32;   /* bf16 mode: keep the residual stream (block outputs,
                            correction tensors) in fp32 storage */
  int32_t conv_impl;     /* 0 = tensor cores wherever the shape allows (stride-1
                            forward and data-gradient convs fed by TMA), 1 = CUDA-core
                            kernels only, 2 = CUDA-core forward + tensor-core gradients,
                            3 = tensor cores with every operand gathered by threads
                            (no TMA producer; same results as 0), 4 = as 0 but the
                            TMA-fed 3x3 convs load one box per tap (no halo tiles;
                            same results as 0) */
  int32_t grad_fp32;     /* bf16 mode: contract gradients (dgrad, wgrad) with fp32
                            operands instead of bf16 ones */
  void* stream;          /* cudaStream_t; NULL = legacy default stream */
  float bn_momentum;     /* rate at which every BN's running statistics follow
                            the batch's in a training forward (the paper states
                            no rule; PyTorch's BatchNorm2d default is 0.1) */
  int32_t inference;     /* 1: plan the forward pass alone for pnn_infer (every BN
                            normalises with its running statistics; activations
                            share buffers, no gradients or optimiser state) */
  int32_t overlap;       /* > 0 (residual correction, N > 1): run the last
                            subnetwork's backward, which needs only D_N (Algorithm
                            2), beside the coarse chain's backward on a second
                            stream, its persistent kernels capped to leave
                            `overlap` SMs to the chain; the chain's term of
                            dL/dx_N is added after both.  0 = phases in sequence */
  int32_t fuse_correction; /* 1 (default): the correction's sums r_j, rt_{j+1},
                            ytilde are formed in the epilogue of the conv that
                            produces their first operand wherever that conv adds
                            a residual (y_j for j < N and rt_N are then not
                            stored; pnn_get_tensor derives them); 0 = launches of
                            their own.  The residual form with overlap > 0 always
                            uses launches of their own. */
} pnn_options;

/* Fill o with the defaults: bf16, residual correction, seed 0, lr 0.1,
 * momentum 0.9, weight decay 5e-4, Nesterov (Section 4), stream_fp32 1,
 * bn_momentum 0.1, inference 0, overlap 0, fuse_correction 1. */
void pnn_default_options(pnn_options* o);

/* Plan the network from a description.  Host only: no GPU work, no device
 * allocation.  *out receives a handle that must be released with pnn_destroy. */
int pnn_create(const pnn_desc* desc, const pnn_options* opts, pnn_net** out);

/* Bytes of device memory the caller must provide. */
int pnn_workspace_bytes(const pnn_net* net, size_t* bytes);

/* Bind a device allocation of at least pnn_workspace_bytes bytes (256-byte
 * aligned).  The caller keeps it alive until pnn_destroy.  Uploads the launch
 * tables and initialises the parameters (He-normal from opts.seed: std
 * sqrt(2/fan_in) for conv and FC weights, BN gamma 1, beta 0, FC bias 0).
 * Synchronises. */
int pnn_bind_workspace(pnn_net* net, void* dev, size_t bytes);

/* Algorithm 1: x (device, batch x in_c x in_h x in_w float32 NCHW), labels
 * (device, batch int32 in [0, classes)).  Writes the mean softmax
 * cross-entropy to loss_dev (device, 1 float; may be NULL).  x and labels
 * must stay valid until pnn_backward returns. */
int pnn_forward(pnn_net* net, const float* x_dev, const int32_t* labels_dev, float* loss_dev);

/* Algorithm 2: gradients of the loss of the preceding pnn_forward with
 * respect to every parameter (eq:etak, eq:phij, eq:deltaj). */
int pnn_backward(pnn_net* net);

/* One SGD step with the gradients of the preceding pnn_backward:
 * d = g + wd*w; v = d (first step) or mu*v + d; w -= lr*(d + mu*v) (Nesterov)
 * or lr*v.  lr <= 0 uses opts.lr. */
int pnn_sgd_step(pnn_net* net, float lr);

/* One whole training step (forward + backward + SGD) replayed from a CUDA
 * graph captured on first use; x_dev/labels_dev as in pnn_forward and must be
 * the same pointers on every call (the graph records them). */
int pnn_train_step(pnn_net* net, const float* x_dev, const int32_t* labels_dev, float* loss_dev);

/* The same step from HOST buffers: copies x and labels to the workspace,
 * runs the step and copies the loss back to *loss_host.  Synchronises. */
int pnn_train_step_host(pnn_net* net, const float* x_host, const int32_t* labels_host, float* loss_host);

/* Wait for the stream and report device-side status words (PNN_ENONFINITE,
 * PNN_ETIMEOUT).  Synchronises. */
int pnn_sync(pnn_net* net);

/* NULL-safe. Does not free the caller's workspace. */
void pnn_destroy(pnn_net* net);

/* ---- parameters (flat vector theta-bar in eq:barf order:
 *      (delta_1, phi_1, ..., delta_N, phi_N, eta_1, ..., eta_{N-1}, eps);
 *      conv weights in (K, C, R, S) order, FC weights (out, in)) ---- */
int pnn_num_params(const pnn_net* net, size_t* n);
int pnn_num_param_tensors(const pnn_net* net, int32_t* n);
/* kind: 0 conv weight, 1 BN gamma, 2 BN beta, 3 FC weight, 4 FC bias;
 * dims[4] (unused trailing dims are 1); offset into theta-bar. */
int pnn_param_tensor_info(const pnn_net* net, int32_t i, int32_t* kind, int32_t dims[4], size_t* offset);
/* Copies of length n (must equal pnn_num_params).  Synchronise. */
int pnn_get_params(pnn_net* net, float* host, size_t n);
int pnn_set_params(pnn_net* net, const float* host, size_t n);
int pnn_get_grads(pnn_net* net, float* host, size_t n);
int pnn_get_momentum(pnn_net* net, float* host, size_t n);

/* ---- interface tensors of the last forward/backward, NCHW float32 ---- */
typedef enum {
  PNN_T_X = 0,      /* x_j = C^j(x), j = 1..N (eq:xjyj) */
  PNN_T_Y = 1,      /* y_j = g^j(x_j), j = 1..N */
  PNN_T_R = 2,      /* r_j = y_j - x_{j+1}, j = 1..N-1 (eq:rk) */
  PNN_T_RTILDE = 3, /* rt_j, j = 1..N (eq:tilderk) */
  PNN_T_YTILDE = 4, /* ytilde (eq:tildey); j ignored */
  PNN_T_D = 5,      /* D_j = dL/drt_j, j = 1..N (Algorithm 2) */
  PNN_T_LOGITS = 6  /* batch x classes; j ignored */
} pnn_tensor;
/* Number of floats of tensor (which, j), or 0 if it does not exist. */
int pnn_tensor_size(const pnn_net* net, int32_t which, int32_t j, size_t* n);
int pnn_get_tensor(pnn_net* net, int32_t which, int32_t j, float* host, size_t n);

/* Per-phase device time of the last eager forward/backward/update in ms,
 * in the paper's column order (Tables gradvgg and grad): pre, fine, coarse,
 * post for forward, the same four for backward, then the SGD update and the
 * total: ms[10]. */
int pnn_get_timings(pnn_net* net, float ms[10]);
/* ---- BN running statistics.  The paper trains with BN and states no rule for
 * them; this library follows PyTorch's BatchNorm2d: every BN layer keeps a
 * running mean (0 at pnn_bind_workspace) and variance (1), and each training
 * forward moves them the fraction opts.bn_momentum towards the batch mean and
 * the unbiased batch variance (n/(n-1) times the biased one, n values per
 * channel).  The delta form's two evaluations of F^j move the same statistics,
 * F^j(x_{j+1}) first.  Layout (host, float): for every BN layer in parameter
 * order (the order of its gamma in the parameter vector), its C running means,
 * then its C running variances.  Get and set synchronise the library stream;
 * n must equal pnn_running_stats_size. */
int pnn_running_stats_size(const pnn_net* net, size_t* n);
int pnn_get_running_stats(pnn_net* net, float* host, size_t n);
int pnn_set_running_stats(pnn_net* net, const float* host, size_t n);

/* ---- inference (Section 3.1's forward, Algorithm 1, in eval mode).  On a net
 * created with opts.inference = 1: x (device, NCHW float32, batch x in_c x
 * in_h x in_w) -> logits (device, batch x classes float32, row-major), every
 * BN normalising with its running statistics (pnn_set_running_stats; a fresh
 * net holds 0 / 1).  Parameters as pnn_set_params.  The pass is captured as a
 * CUDA graph on the first call for a given (x, logits) pair and replayed after
 * that (with profiling enabled, pnn_profile, it runs eagerly so that every
 * launch is timed); it runs asynchronously on the library stream (pnn_sync
 * waits).
 * PNN_ESTATE on a training net; pnn_forward, pnn_backward, pnn_sgd_step,
 * pnn_train_step, pnn_time_phases and the gradient accessors return PNN_ESTATE
 * on an inference net, and pnn_get_tensor gives only PNN_T_LOGITS there. */
int pnn_infer(pnn_net* net, const float* x, float* logits);

/* ---- tearing (Section 4.2, the remark after Table grad: a decomposition of the
 * body into subnetworks of equal computational cost rather than equal numbers
 * of RUs).  Both calls are host-only and need no GPU. */
typedef enum { PNN_COST_FLOPS = 0, PNN_COST_BYTES = 1 } pnn_cost_kind;
/* Cost of each of the n = desc->n_body layers of the block-repetitive part g
 * in the untorn network (desc's body as one segment, no coarse network): the
 * algorithmic FLOPs (conv FLOPs = 2 * B*P*Q*K*C*R*S over the layer's forward,
 * data-gradient and weight-gradient convolutions) or HBM bytes (each operand
 * read once, each result written once, as pnn_profile_read counts them) of the
 * layer's forward and backward ops under opts (NULL: defaults).  desc->segments
 * and the coarse fields are ignored.  out: caller-owned, n doubles. */
int pnn_block_costs(const pnn_desc* desc, const pnn_options* opts, int32_t kind, double* out, int32_t n);
/* Cut n layers with costs cost[0..n-1] (finite, >= 0) into n_seg consecutive
 * non-empty segments whose largest cost sum is as small as possible (exact).
 * Among the optimal cuts it returns the one whose segments, from the first on,
 * each take as many layers as the optimum allows.  segments: caller-owned,
 * n_seg ints (layers per segment, summing to n).  Time O(n_seg * n^2);
 * PNN_EINVAL unless 1 <= n_seg <= n and n_seg * n^2 <= 4e9. */
int pnn_partition(const double* cost, int32_t n, int32_t n_seg, int32_t* segments);

/* Per-phase device time of whole training steps replayed from CUDA graphs,
 * in the order of pnn_get_timings (ms[10]): each phase (pre, fine, coarse,
 * post forward; post, coarse, fine, pre backward; update) is captured as its
 * own graph and bracketed by events on the library stream, and the times are
 * the mean over `steps` steps.  The phases of Tables gradvgg and grad, without
 * the launch gaps of an eager step.  x and labels are device pointers as for
 * pnn_train_step; each step updates the parameters.  A network that has not
 * stepped yet first takes one untimed eager step (it initialises the momentum
 * buffers), so it then takes steps + 1 steps in all.  Synchronises the library
 * stream.  PNN_ESTATE while profiling is enabled; PNN_EINVAL for steps <= 0. */
int pnn_time_phases(pnn_net* net, const float* x, const int32_t* labels, int32_t steps, float ms[10]);
/* Counts of the step's kernel launches: forward, backward, update. */
int pnn_launch_counts(const pnn_net* net, int32_t counts[3]);

/* ---- profiling: with enable != 0 every kernel launch of eager calls
 * (pnn_forward / pnn_backward / pnn_sgd_step) is bracketed by CUDA events on
 * the library stream; pnn_profile_read synchronises, folds the recorded
 * launches into per-kind totals and returns, for one kernel kind, the summed
 * device time (ms), the launch count and the algorithmic FLOPs and bytes of
 * those launches (conv FLOPs = 2 * B*P*Q*K*C*R*S; bytes = each operand read
 * once and each result written once).  Enabling or disabling resets totals
 * and drops a captured step graph.  Kinds are 0 .. pnn_num_kernel_kinds()-1. */
int pnn_profile(pnn_net* net, int32_t enable);
int pnn_profile_read(pnn_net* net, int32_t kind, double* ms, int64_t* launches, double* flops, double* bytes);

/* One record per kernel launch bracketed since pnn_profile(net, 1), in launch
 * order: kind (as for pnn_kernel_kind_name), variant (tensor-core convs:
 * 0 = operands gathered by threads, 1 = fed by TMA, 2 = fed by TMA with the
 * wide epilogue of one-k-step tiles, 3 = fed by TMA with halo tiles),
 * step phase (0 preprocessing
 * forward, 1 fine forward, 2 coarse forward, 3 head forward, 4 head backward,
 * 5 coarse backward, 6 correction backward, 7 fine backward, 8
 * preprocessing backward), the number of layer instances grouped in the
 * launch and its work items (tiles or rows), the first instance's shape
 * (convolutions: C_in, C_out, kernel size, stride, H_out, W_out; other kinds:
 * C, H, W of the tensor read, then zeros), device time and algorithmic
 * FLOPs and bytes as for pnn_profile_read.  Writes min(max, recorded)
 * records to out (caller-owned host memory) and the number recorded to
 * *count; synchronises the library stream.  Records stay until the next
 * pnn_profile call. */
typedef struct pnn_trace {
  int32_t kind, variant, phase, instances, tiles;
  int32_t shape[6];
  int32_t block; /* fine-wave launches (phases 1 and 7): the layer's position
                    in its segment, its index in g for an untorn network
                    (n_seg = 1); -1 for every other launch */
  double ms, flops, bytes;
} pnn_trace;
int pnn_profile_trace(pnn_net* net, int32_t max, pnn_trace* out, int32_t* count);
int32_t pnn_num_kernel_kinds(void);
const char* pnn_kernel_kind_name(int32_t kind); /* NULL for a bad kind */

/* Debug builds (compiled with PNN_DEBUG_CHECKS): the first misaligned vector
 * access a tensor-core kernel detected and skipped, as (source line << 40 |
 * address low 40 bits); 0 if none or in release builds. */
uint64_t pnn_debug_word(void);

/* ---- one grouped convolution on caller buffers ----
 * The three contractions of a training step's convolution layers (Section 3.2:
 * Algorithm 1's forward g^j, Algorithm 2's data and weight gradients), run
 * alone through the same tensor-core kernels pnn_forward / pnn_backward
 * launch, so that each kernel can be checked element by element.  n instances
 * (each its own geometry and buffers) form one grouped launch, as the N
 * subnetworks' layers do in a step.  Zero padding ksize/2; p = (h + 2*pad -
 * ksize)/stride + 1, q likewise.  Contraction operands are rounded to bf16
 * (round to nearest even), products accumulate in fp32.
 *   mode PNN_CONV_FORWARD  y[n][p][q][kk] = res + sum_{r,s,cc} v(x)[n][p*stride+r-pad][q*stride+s-pad][cc] * w[kk][r][s][cc]
 *                          with v(x) = bn_scale[cc]*x + bn_shift[cc], then max(0, .) when
 *                          relu != 0, when bn_scale is given (the BN(+ReLU) of the layer
 *                          before, applied on load), else v(x) = x; y rounded to y_dtype.
 *                          y_mean / y_rstd (optional, device, k floats): the batch
 *                          statistics of y that a following BN layer uses (mean, 1/sqrt(var + 1e-5),
 *                          biased variance over batch*p*q rows, Section 4's BN)
 *   mode PNN_CONV_DGRAD    dx[n][i][j][cc] (+)= sum_{r,s,kk} dy[n][p][q][kk] * w[kk][r][s][cc]
 *                          over the (p, q) with p*stride+r-pad = i, q*stride+s-pad = j.
 *                          With bn_mean / bn_rstd given (x = the BN input h, bn_scale /
 *                          bn_shift / relu its forward BN): dbeta[cc] = sum g and dgamma[cc] =
 *                          sum g * (h - mean) * rstd over all rows, g = dx masked by the ReLU of
 *                          bn_scale*h + bn_shift (the BN-backward sums of that layer)
 *   mode PNN_CONV_WGRAD    dw[kk][r][s][cc] = sum_{n,p,q} dy[n][p][q][kk] * v(x)[n][p*stride+r-pad][q*stride+s-pad][cc]
 * impl: 0 = the kernel a training step would choose, 1 = the TMA-fed kernel
 * (stride 1 only; PNN_EINVAL where the shape does not allow it), 2 = the
 * thread-gathered kernel, 3 = the TMA-fed kernel with one box per 3x3 tap
 * (1 and 0 use one halo box per 128-pixel tile where the tile lies inside
 * one image: 3x3, 128 | h*w, w <= 63, 16 | the A source's channels <= 64).  c and k multiples of 8.  All pointers are device
 * memory of the current device, NHWC with the batch folded into the rows;
 * w is bf16 [k][ksize][ksize][c].  The caller owns every buffer and a
 * workspace of pnn_conv_workspace_bytes bytes (256-byte aligned); the call
 * allocates nothing, enqueues on `stream` (NULL = legacy default) and
 * synchronises it.  Errors: PNN_EINVAL, PNN_ENOMEM (workspace too small),
 * PNN_ECUDA, PNN_ETIMEOUT; message in pnn_last_error(NULL). */
typedef enum { PNN_CONV_FORWARD = 0, PNN_CONV_DGRAD = 1, PNN_CONV_WGRAD = 2 } pnn_conv_mode;
typedef enum { PNN_DT_F32 = 0, PNN_DT_BF16 = 1 } pnn_dtype;
typedef struct pnn_conv_args {
  int32_t batch, h, w, c;        /* input geometry */
  int32_t k, ksize, stride;      /* output channels, 1 or 3, 1 or 2 */
  const void* x;                 /* forward / weight gradient input; data gradient: BN input (optional) */
  int32_t x_dtype;               /* pnn_dtype */
  const float* bn_scale;         /* optional, c floats: read v(x) instead of x */
  const float* bn_shift;
  int32_t relu;
  const void* wt;                /* bf16 weights [k][ksize][ksize][c] */
  void* y;                       /* forward output, batch*p*q x k */
  int32_t y_dtype;
  const void* res;               /* forward: optional residual added before rounding, batch*p*q x k */
  int32_t res_dtype;
  float* y_mean;                 /* forward: optional batch statistics of y, k floats each */
  float* y_rstd;
  const float* dy;               /* gradients: float32, batch*p*q x k */
  float* dx;                     /* data gradient output, batch*h*w x c float32 */
  int32_t accumulate;            /* data gradient: add into dx instead of overwriting it */
  const float* bn_mean;          /* data gradient: optional BN-backward sums (see above) */
  const float* bn_rstd;
  float* dgamma;
  float* dbeta;
  float* dw;                     /* weight gradient output, k x ksize x ksize x c float32 */
} pnn_conv_args;
int pnn_conv_workspace_bytes(int32_t mode, int32_t impl, int32_t n, const pnn_conv_args* args, size_t* bytes);
int pnn_conv_run(int32_t mode, int32_t impl, int32_t n, const pnn_conv_args* args, void* workspace,
                 size_t workspace_bytes, void* stream);
/* pnn_conv_run, then `repeat` (> 0) further launches of the convolution
 * kernel alone between two CUDA events on `stream` (each rewrites what the
 * first wrote; accumulate must be 0): *ms_per_launch = their mean device
 * time.  A microbenchmark of one grouped launch; same errors as pnn_conv_run. */
int pnn_conv_time(int32_t mode, int32_t impl, int32_t n, const pnn_conv_args* args, void* workspace,
                  size_t workspace_bytes, void* stream, int32_t repeat, float* ms_per_launch);

/* ---- allocation-free weight gradient of one convolution ----
 * The paper has no counterpart to this call.  It exists for callers that
 * cannot allocate device memory at the point they need the result, e.g.
 * code running inside a memory pool they do not control, or a runtime that
 * forbids cudaMalloc after start-up.  It computes the same weight gradient
 * as the tensor-core kernel pnn_backward uses,
 *   dw[kk][r][s][cc] = sum_{n,p,q} dy[n][p][q][kk] * x[n][p*stride+r-pad][q*stride+s-pad][cc]
 * (pad = ksize/2, zero padding, both operands rounded to bf16, fp32
 * accumulation), but keeps its split-K partial sums, launch descriptors and
 * status word in fixed-size device arrays compiled into the library: 16 MiB
 * of partial sums, so k * ksize * ksize * c must not exceed 4,194,304
 * (PNN_EINVAL otherwise).  It calls no cudaMalloc, cudaFree or allocating
 * library routine.
 *   x   device, batch x h x w x c float32, NHWC
 *   dy  device, batch x p x q x k float32, NHWC, p = (h + 2*pad - ksize)/stride + 1
 *   dw  device, k x ksize x ksize x c float32 (written, not accumulated)
 *   c and k multiples of 8; ksize 1 or 3; stride 1 or 2; stream NULL = legacy default.
 * Every GPU that loads the library keeps these arrays until the process ends.
 * The first call on a device looks up their device addresses (once per
 * device, thread-safe).  All calls share the arrays and each call overwrites them: calls that
 * overlap on the GPU (other streams, other threads) race.  Synchronises.
 * Errors: PNN_EINVAL (arguments), PNN_ECUDA, PNN_ETIMEOUT; message in
 * pnn_last_error(NULL). */
int pnn_conv_wgrad_noalloc(const float* x, const float* dy, float* dw, int32_t batch, int32_t h, int32_t w,
                           int32_t c, int32_t k, int32_t ksize, int32_t stride, void* stream);

/* Failure-detection self-test (no counterpart in the paper).  Every device
 * wait of the library's kernels is bounded: on expiry a kernel records status
 * 3, releases what it holds and returns, and the host reports PNN_ETIMEOUT.
 * This call exercises that path on purpose: it launches one thread that
 * arrives once on an mbarrier expecting two arrivals and waits on it with the
 * kernels' bounded wait, limited to limit_ns (0 < limit_ns <= 1e10).  The
 * phase never completes, so the call returns PNN_ETIMEOUT after about
 * limit_ns, and the CUDA context stays usable.  stream: cudaStream_t (NULL =
 * legacy default stream); synchronises it.  Allocates nothing. */
int pnn_selftest_wait_timeout(int64_t limit_ns, void* stream);

const char* pnn_last_error(const pnn_net* net);
const char* pnn_status_string(int status);

#ifdef __cplusplus
}
#endif
#endif /* PNN_H_ */
