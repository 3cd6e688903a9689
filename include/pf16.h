/*
 * pf16 -- pure-FP16 ResNet-50 training kernels for NVIDIA GB300 (sm_103a).
 *
 * The library implements the hot path of "Distributed low-precision Training
 * Without Mixed Precision" (arXiv 1911.07384): ResNet-50 trained with every
 * activation, weight and gradient stored in IEEE binary16 and every
 * arithmetic operation done in binary16, with no FP32 master copy of any
 * parameter (Sec. 5.2) and with the x0.25 scaling after each BatchNorm of a
 * residual block (Sec. 4.2).  Convolutions accumulate in FP16 inside the
 * tensor cores (tcgen05, FP16 accumulators in tensor memory).
 *
 * Conventions shared by every entry point
 *  - Tensors are dense binary16 bit patterns (uint16_t) in DEVICE memory,
 *    owned and allocated by the caller.  Activations are NHWC (C innermost),
 *    convolution weights KRSC.  Every tensor pointer must be 16-byte aligned.
 *  - Calls are asynchronous and stream-ordered on `stream` (a cudaStream_t;
 *    NULL = the legacy default stream).  The library never allocates or frees
 *    memory and keeps no tensors between calls; scratch memory is the
 *    caller's `ws` buffer, sized by the matching *_workspace_size function.
 *    Calls on distinct streams may run concurrently; calls that share a
 *    workspace must be ordered by the caller.
 *  - Every argument is validated on the host before anything is launched; an
 *    invalid call returns a negative status and launches nothing.
 *  - Device-side waits are bounded; one that runs out records PF16_ERR_TIMEOUT
 *    in a device status word, read (and cleared) by pf16_sync_status.
 *  - Rounding: IEEE roundTiesToEven for every binary16 operation, subnormals
 *    kept (no flush to zero), never a fused multiply-add unless stated.
 */
#ifndef PF16_H
#define PF16_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---------------------------------------------------------------- status */
enum {
  PF16_OK = 0,
  PF16_ERR_NULL = -1,        /* a required pointer is NULL */
  PF16_ERR_ALIGN = -2,       /* a tensor pointer is not 16-byte aligned */
  PF16_ERR_SHAPE = -3,       /* non-positive, inconsistent or too-large sizes */
  PF16_ERR_UNSUPPORTED = -4, /* well-formed but outside what the kernels cover */
  PF16_ERR_WORKSPACE = -5,   /* workspace NULL or smaller than required */
  PF16_ERR_CUDA = -6,        /* a CUDA runtime or driver call failed */
  PF16_ERR_TIMEOUT = -7,     /* a bounded device-side wait expired */
  PF16_ERR_ARG = -8          /* invalid flag, phase or enum value */
};

/* ----------------------------------------------------------------- flags */
#define PF16_ACCUMULATE 0x1u  /* conv: out = rn(out + result) instead of out = result */
#define PF16_F32_ACCUM 0x4u   /* conv: FP32 accumulation in the tensor core, each output rounded once
                                 to FP16 -- a contrast to the paper's pure-FP16 method (Sec. 1, 2:
                                 the mixed-precision accumulation it does without), not part of it */
#define PF16_BN_RELU 0x1u     /* BN: apply ReLU to the output */
#define PF16_BN_RESIDUAL 0x2u /* BN: add the residual tensor before the ReLU */
#define PF16_BN_SWAP 0x4u     /* BN, with PF16_BN_RESIDUAL: the "swap" variant of a block's last
                                 BatchNorm (Sec. 4.1): y = gamma*(s*xhat + residual) + beta */

/* ------------------------------------------------------------ convolution
 * Convolution of the ResNet-50 layers (Sec. 5.1) in pure FP16 (Sec. 5.2):
 * dilation 1, one group, the same stride and padding on both axes.
 *   x  [n][h][w][c]    input activations (NHWC)
 *   w  [k][r][s][c]    weights (KRSC)
 *   y  [n][p][q][k]    output, p = (h + 2 pad - r)/stride + 1, q likewise
 * Supported: c and k multiples of 64 (any n, h, w), or c == 3 with k == 64
 * (the ResNet-50 stem; its 7x7 patches are staged through the workspace),
 * or h == w == r == s == 1 with c a multiple of 64 and k a multiple of 8
 * (the fully connected layer).  r, s <= 7; stride 1 or 2; pad < r. */
typedef struct {
  int32_t n, h, w, c, k, r, s, stride, pad;
} pf16_conv_desc;

#define PF16_PASS_FWD 0
#define PF16_PASS_DGRAD 1
#define PF16_PASS_WGRAD 2

/* Bytes of workspace the given pass needs (0 if none).  Returns 0 for an
 * invalid descriptor as well; the call then reports the error. */
size_t pf16_conv_workspace_size(const pf16_conv_desc* d, int pass);

/* Forward: y[n,p,q,k] = sum_{r,s,c} x[n, p*st+r-pad, q*st+s-pad, c] * w[k,r,s,c]
 * (zero outside x).  FP16 products, FP16 accumulation in the tensor core,
 * FP16 result.  flags: PF16_ACCUMULATE, PF16_F32_ACCUM (the contrast variant:
 * products accumulated in FP32 inside the tensor core, one rounding to FP16). */
int pf16_conv_fwd(const pf16_conv_desc* d, const uint16_t* x, const uint16_t* w, uint16_t* y,
                  void* ws, size_t ws_bytes, uint32_t flags, void* stream);

/* Forward with the BatchNorm statistics of its output (Eq. 1, Sec. 4.2:
 * every conv of ResNet-50 but the FC layer feeds a BatchNorm).  Same
 * arguments and result as pf16_conv_fwd with flags 0, and in addition each
 * epilogue warp of the GEMM reduces the output rows it stores into a running
 * (mean, biased variance, count) per output channel -- FP16 halving trees
 * over 32 rows merged by the count-aware parallel-variance rule -- written to
 * `stats` (stats_bytes >= pf16_conv_bnstats_size(d), 16-byte aligned,
 * caller-owned; no initial contents needed).  pf16_bn_fwd_bwd phase 0 takes
 * it through pf16_bn_tensors.conv_stats and skips its own statistics pass
 * over y.  k must be a multiple of 64 (PF16_ERR_UNSUPPORTED otherwise). */
size_t pf16_conv_bnstats_size(const pf16_conv_desc* d);
int pf16_conv_fwd_bnstats(const pf16_conv_desc* d, const uint16_t* x, const uint16_t* w, uint16_t* y,
                          void* ws, size_t ws_bytes, void* stats, size_t stats_bytes, void* stream);

/* Data gradient: dx[n,h,w,c] = sum over the (k,r,s) with h+pad-r = p*st and
 * w+pad-s = q*st in range of dy[n,p,q,k] * w[k,r,s,c]; stride 2 is split into
 * its stride-phase sub-problems, so no zero-insertion work is done.  Every
 * element of dx is written (zeros included) unless PF16_ACCUMULATE, in which
 * case dx = rn(dx + result) and positions no tap reaches are left unchanged.
 * PF16_F32_ACCUM as for the forward.
 * Not available for c == 3 (the stem needs no input gradient). */
int pf16_conv_dgrad(const pf16_conv_desc* d, const uint16_t* dy, const uint16_t* w, uint16_t* dx,
                    void* ws, size_t ws_bytes, uint32_t flags, void* stream);

/* Data gradient with the backward statistics of the BatchNorm whose output
 * gradient it is (Eq. 1-2 differentiated; the backward counterpart of
 * pf16_conv_fwd_bnstats).  dx, the result, is dL/dy of a BatchNorm described
 * by `bn`: its input x (n x h x w x c, the conv output its forward normalised),
 * its ReLU bit mask (as written by pf16_bn_fwd_bwd phase 0; NULL for a
 * BatchNorm without ReLU) and its saved mean and invstd.  Same arguments and
 * dx as pf16_conv_dgrad with flags 0; in addition each epilogue warp of the
 * GEMM reduces, per channel, dy' = dx where the ReLU passed and dy' * xhat,
 * xhat = rn(rn(x - mean) * invstd), over the 32 rows of each tile it stores:
 * FP16 pairwise sums, zero leaves for rows past the tensor, pushed into the
 * warp's tree of tiles, which is padded with zero leaves to a power of two.
 * The CTAs' nodes go to `stats` (stats_bytes >= pf16_conv_dgrad_bnstats_size(d),
 * 16-byte aligned, caller-owned, no initial contents needed);
 * pf16_bn_fwd_bwd phase 1 takes it through pf16_bn_tensors.conv_stats and
 * skips its statistics pass over dy and x.  Requires c a multiple of 64 and
 * either stride 1 or a stride-2 filter larger than 1x1 whose four stride
 * phases all receive taps and share their output grid and first dy row and
 * column (for 3x3 with pad 1: even h and w, as in ResNet; the phases then run
 * as one GEMM whose rows land at scattered pixels, and the warps' rows are
 * those rows);
 * PF16_ERR_UNSUPPORTED otherwise, and the size function then returns 0.
 * x, mean, invstd 16-byte aligned, relu_mask 8-byte aligned. */
typedef struct {
  const uint16_t* x;         /* the BatchNorm's input, n x h x w x c */
  const uint8_t* relu_mask;  /* its ReLU decisions (bit mask), or NULL: no ReLU */
  const uint16_t* mean;      /* its saved mean [c] */
  const uint16_t* invstd;    /* its saved invstd [c] */
} pf16_bn_source;
size_t pf16_conv_dgrad_bnstats_size(const pf16_conv_desc* d);
int pf16_conv_dgrad_bnstats(const pf16_conv_desc* d, const uint16_t* dy, const uint16_t* w, uint16_t* dx,
                            void* ws, size_t ws_bytes, const pf16_bn_source* bn, void* stats,
                            size_t stats_bytes, void* stream);

/* pf16_conv_dgrad_bnstats plus an addend: dx = rn(result + a), a = add where
 * add_mask's bit is set (the layout of pf16_bn_desc's relu_mask for a
 * n x h x w x c tensor) and +0 elsewhere; NULL add_mask: a = add.  The
 * statistics are those of this dx.  This is the gradient at the input of an
 * identity-shortcut residual block (Sec. 4.2): the shortcut's share (the
 * block's output gradient where its final ReLU passed, add and add_mask) plus
 * the first convolution's data gradient, and it is the output gradient of the
 * previous block's last BatchNorm (bn).  dx is bit-identical to that
 * BatchNorm's dresidual followed by pf16_conv_dgrad with PF16_ACCUMULATE;
 * the residual BatchNorm's backward then needs no dresidual output.
 * Requires a 1x1 filter with stride 1 and pad 0 and c a multiple of 64
 * (PF16_ERR_UNSUPPORTED); add is n x h x w x c, 16-byte aligned, and must not
 * overlap dx (PF16_ERR_ARG); add_mask 8-byte aligned. */
int pf16_conv_dgrad_bnstats_add(const pf16_conv_desc* d, const uint16_t* dy, const uint16_t* w, uint16_t* dx,
                                void* ws, size_t ws_bytes, const pf16_bn_source* bn, const uint16_t* add,
                                const uint8_t* add_mask, void* stats, size_t stats_bytes, void* stream);

/* Weight gradient: dw[k,r,s,c] = sum_{n,p,q} dy[n,p,q,k] * x[n, p*st+r-pad, q*st+s-pad, c].
 * The reduction over n*p*q pixels is split into chunks, each accumulated in
 * FP16 by the tensor core into FP16 partials in the workspace, which are then
 * summed by a balanced pairwise FP16 tree.  flags: 0 or PF16_F32_ACCUM (each
 * chunk accumulated in FP32 and rounded once to its FP16 partial; the tree
 * stays FP16); PF16_ERR_ARG otherwise. */
int pf16_conv_wgrad(const pf16_conv_desc* d, const uint16_t* x, const uint16_t* dy, uint16_t* dw,
                    void* ws, size_t ws_bytes, uint32_t flags, void* stream);

/* ----------------------------------------- BatchNorm in the operand path
 * A conv whose input is the output of a BatchNorm (Eq. 1, Eq. 2, x post_scale
 * of Sec. 4.2, optional ReLU) can take the BatchNorm's INPUT x and apply it
 * to each operand tile in shared memory, between the tile's arrival and the
 * tensor core's read -- the same FP16 op sequence as pf16_bn_fwd_bwd's apply
 * (xhat = rn(rn(x - mean) * invstd); z = rn(rn(rn(gamma * xhat) + beta) *
 * post_scale); ReLU), so the conv sees bit for bit the operand it would read
 * from the stored BatchNorm output, and its result is bit-identical to
 * pf16_bn_fwd_bwd phase 0 followed by the plain call.  The BatchNorm output
 * is then never written: phase 0 runs with y = NULL (statistics only) and the
 * convs that read the output take the input instead.
 * mean, invstd: the BatchNorm's saved statistics (phase 0); gamma, beta: its
 * parameters; all [c], 16-byte aligned.  flags: PF16_BN_RELU or 0. */
typedef struct {
  const uint16_t* mean;
  const uint16_t* invstd;
  const uint16_t* gamma;
  const uint16_t* beta;
  uint16_t post_scale;  /* binary16 bits */
  uint32_t flags;       /* PF16_BN_RELU or 0 */
  uint8_t* relu_mask;   /* pf16_conv_fwd_bnin only, optional (needs PF16_BN_RELU): the ReLU decisions,
                           written in pf16_bn_fwd_bwd's bit-mask layout (any alignment) */
} pf16_bn_operand;

/* Forward conv of x' = BN(x) (x: the BatchNorm's input, n x h x w x c):
 * y as pf16_conv_fwd of x', and, with a non-NULL stats buffer, the
 * statistics of y as pf16_conv_fwd_bnstats.  Covers the dense 1x1 / stride 1
 * / pad 0 layers (a bottleneck's last conv); other shapes return
 * PF16_ERR_UNSUPPORTED.  No workspace. */
int pf16_conv_fwd_bnin(const pf16_conv_desc* d, const uint16_t* x, const pf16_bn_operand* bn, const uint16_t* w,
                       uint16_t* y, void* stats, size_t stats_bytes, void* stream);
/* Weight gradient of the same layer from x' = BN(x): dw as pf16_conv_wgrad
 * of x' (flags 0; the same workspace).  bn->relu_mask must be NULL.  Same
 * shape coverage as pf16_conv_fwd_bnin. */
int pf16_conv_wgrad_bnin(const pf16_conv_desc* d, const uint16_t* x, const pf16_bn_operand* bn, const uint16_t* dy,
                         uint16_t* dw, void* ws, size_t ws_bytes, void* stream);

/* Weight gradient without any caller workspace (the paper has no counterpart:
 * this is a convenience of the library).  Same arguments, result and error
 * codes as pf16_conv_wgrad, minus ws / ws_bytes.  It is meant for callers that
 * cannot give the library scratch memory: hosts that plan all device memory
 * themselves and do not let a library request more, deployments that forbid
 * device allocation after set-up, or bindings with no CUDA allocator at hand;
 * it also spares a training loop the device-wide stall a cudaMalloc can cause.
 * Its split-K scratch is one fixed array of PF16_WGRAD_NOALLOC_SCRATCH_BYTES
 * compiled into the library; every device that loads it keeps the array until
 * the process exits.  Nothing is allocated or freed by the call.
 *  - A layer whose split-K scratch (pf16_conv_workspace_size(d,
 *    PF16_PASS_WGRAD)) exceeds the array is rejected with PF16_ERR_WORKSPACE
 *    before anything is launched; this includes the c == 3 stem, whose patch
 *    buffer is far larger.  Every other ResNet-50 layer at batch 256 fits.
 *  - The first call on each device looks up the array's device address (with
 *    that device current); make that first call before any stream capture.
 *    The address is kept for the life of the process: after cudaDeviceReset
 *    on a device this entry point must not be called on that device again.
 *  - All calls share the one array, which keeps the last call's contents
 *    (no call depends on them).  Calls that can overlap on the GPU -- on
 *    different streams, or on one device from several threads -- race on it;
 *    order them on one stream or use pf16_conv_wgrad with separate workspaces. */
#define PF16_WGRAD_NOALLOC_SCRATCH_BYTES (32u << 20)
int pf16_conv_wgrad_noalloc(const pf16_conv_desc* d, const uint16_t* x, const uint16_t* dy,
                            uint16_t* dw, uint32_t flags, void* stream);

/* ------------------------------------------------------------------- SGD
 * One step of SGD with momentum and coupled weight decay, the PyTorch
 * ImageNet recipe the paper adopts (Sec. 5.1), done entirely in FP16 with no
 * master copy (Sec. 5.2).  In place on w[n] and v[n] (the momentum buffer,
 * start it at +0), gradient g[n]; lr, momentum and wd are binary16 bit
 * patterns.  Per element, each op rounded once to binary16, no FMA:
 *   g' = rn(g + rn(wd*w))   (skipped entirely when wd is +0)
 *   v  = rn(rn(momentum*v) + g')
 *   w  = rn(w - rn(lr*v))
 * flags must be 0.  n may be 0 (nothing is launched). */
int pf16_sgd_update(uint16_t* w, uint16_t* v, const uint16_t* g, size_t n, uint16_t lr,
                    uint16_t momentum, uint16_t wd, uint32_t flags, void* stream);

/* ------------------------------------------------- data-parallel exchange
 * The combining step of the fixed-order FP16 gradient all-reduce of
 * data-parallel training (Sec. 5.1: ResNet-50 on 8 to 128 GPUs, each with
 * its own batch and its own BatchNorm statistics, their gradients averaged
 * before every SGD step; Sec. 5.2: that average is taken in FP16 too).
 * `planes` holds `world` gradient planes of n binary16 values, plane r at
 * planes + r * plane_stride (elements) -- the same slice of every rank's
 * gradient, in rank order.  Per element i:
 *   out[i] = rn(T(i) * scale),  T(i) = the perfect pairwise tree over the
 *   leaves planes[0][i], ..., planes[world-1][i], padded with +0 leaves to
 *   the next power of two, each node rn(left + right)
 * with scale normally rn(1/world) (binary16 bits; the multiply is skipped
 * when scale is 0x3C00 = 1).  The sum comes before the scaling so that small
 * gradients keep their low bits (a scale of 1/128 first would push them 7
 * binades toward underflow); it overflows only where the sum of the world's
 * gradients exceeds 65,504.  The order depends only on world and i, so every
 * rank that combines the same planes gets the same bits, whatever the
 * launch configuration.
 * n and plane_stride are multiples of 8, plane_stride >= n, 1 <= world <=
 * 1024; out may be planes itself (plane 0 is overwritten only after every
 * plane of an element was read) and must not overlap the other planes.
 * n == 0 launches nothing.  Errors: PF16_ERR_NULL, PF16_ERR_ALIGN (16-byte
 * alignment), PF16_ERR_SHAPE. */
int pf16_allreduce_combine(const uint16_t* planes, int32_t world, size_t n, size_t plane_stride,
                           uint16_t scale, uint16_t* out, void* stream);

/* ------------------------------------------------------------- BatchNorm
 * BatchNorm with batch statistics over the n*h*w rows of each of c channels
 * (Eq. 1, Eq. 2), each output then multiplied by post_scale (0x3400 = 0.25
 * inside residual blocks, 0x3C00 = 1 for the stem, Sec. 4.2), optionally
 * plus a residual tensor and followed by ReLU (flags).  All arithmetic FP16,
 * and no forward partial result can overflow unless the data do: the
 * forward mean and biased variance are balanced pairwise trees of (mean, mean
 * squared deviation) nodes merged by the parallel-variance rule with exact
 * counts (equal counts: mean node rn(a/2 + rn(b/2)), one fused multiply-add).
 * The backward sums of dy' and dy'*xhat are pairwise trees of rn(a + b) over
 * zero-padded power-of-two leaves -- gradients are small, and a halving node
 * would drop the low bits of subnormal partial means -- giving dbeta =
 * rn(s * sum dy') and dgamma = rn(s * sum dy'*xhat), and the means
 * rn(rn(sum * rn(2^L/R)) * 2^-L), L = ceil(log2 R).
 * The tree shapes depend only on n*h*w and c.
 *   phase 0 (forward, training):  reads x, gamma, beta[, residual];
 *       writes y, mean, invstd (per channel, saved for the backward).
 *       y may be NULL: then only mean and invstd are computed (relu_mask
 *       must be NULL too), for a conv that applies this BatchNorm in its
 *       operand path (pf16_conv_fwd_bnin).
 *       With PF16_BN_RELU and a non-NULL relu_mask it also writes the ReLU
 *       decisions: n*h*w*c/8 bytes, bit j of byte [row*(c/8) + g] set iff
 *       output channel 8g+j of that row is > 0 (so y > 0).  Any alignment.
 *   phase 1 (backward): reads x, gamma, mean, invstd, dy and, with
 *       PF16_BN_RELU, the ReLU decisions: from relu_mask when it is non-NULL
 *       (as written by phase 0; y_saved is then not read and may be NULL),
 *       else from y_saved (y > 0).  Writes dx, dgamma, dbeta and, if
 *       non-NULL, dresidual (= dy masked by ReLU, the gradient flowing to the
 *       residual input).  Both sources give bit-identical results; the mask
 *       moves 1/16 of the bytes.
 *   PF16_BN_SWAP (with PF16_BN_RESIDUAL; Sec. 4.1's switch, off in the
 *       paper's best runs): the forward is y = gamma * (s*xhat + residual) +
 *       beta [, ReLU]; the backward also reads residual and gives dbeta =
 *       sum dy', dgamma = rn(rn(s * sum dy'*xhat) + sum dy'*residual) (a second
 *       statistics pass) and dresidual = gamma * dy'; dx is unchanged in form.
 *       conv_stats is not accepted in its phase 1 (PF16_ERR_UNSUPPORTED).
 * relu_mask is ignored without PF16_BN_RELU (the bit mask is a storage
 * choice of this library, not part of the paper's method).
 * conv_stats (optional, 16-byte aligned):
 *   phase 0: when x is the output of a pf16_conv_fwd_bnstats call that filled
 *       this buffer (and nothing has written x or the buffer since), the mean
 *       and variance are taken from its partial statistics instead of a pass
 *       over x;
 *   phase 1: when dy is the output of a pf16_conv_dgrad_bnstats call that
 *       filled this buffer for this BatchNorm (same x, mask, mean, invstd),
 *       the means of dy' and dy'*xhat (and dgamma, dbeta) come from its
 *       partial trees instead of a pass over dy and x;
 *   either way the result is the same BatchNorm up to the FP16 rounding of a
 *   different reduction tree.
 * c must be a multiple of 8 and at most 2048. */
typedef struct {
  int32_t n, h, w, c;
  uint16_t eps;        /* binary16 bits, e.g. 0x00A8 (1e-5, subnormal) */
  uint16_t post_scale; /* binary16 bits */
  uint32_t flags;      /* PF16_BN_RELU | PF16_BN_RESIDUAL */
} pf16_bn_desc;

typedef struct {
  const uint16_t *x, *gamma, *beta, *residual, *dy, *y_saved;
  uint16_t *y, *mean, *invstd, *dx, *dgamma, *dbeta, *dresidual;
  uint8_t* relu_mask; /* optional ReLU bit mask: written by phase 0, read by phase 1 */
  const void* conv_stats; /* optional: partial statistics from pf16_conv_fwd_bnstats (phase 0)
                             or pf16_conv_dgrad_bnstats (phase 1) */
} pf16_bn_tensors;

size_t pf16_bn_workspace_size(const pf16_bn_desc* d);
int pf16_bn_fwd_bwd(const pf16_bn_desc* d, int phase, const pf16_bn_tensors* t, void* ws,
                    size_t ws_bytes, void* stream);

/* The stem's BatchNorm with ReLU and the 3x3 / stride 2 / pad 1 max pooling
 * that follows it in one call (Sec. 5.1's ResNet-50 stem): phase 0 of
 * pf16_bn_fwd_bwd (flags exactly PF16_BN_RELU: no residual; conv_stats as
 * there) whose output y goes straight into the pooling, so y is never
 * stored (t->y must be NULL).  Writes t->mean, t->invstd, t->relu_mask (if
 * non-NULL, as phase 0) and pooled[n][p][q][c], argmax[n][p][q][c] as
 * pf16_maxpool_fwd_argmax (p < (h - 1) / 2 + 1, q < (w - 1) / 2 + 1).  The
 * results are bit for bit those of pf16_bn_fwd_bwd(phase 0) followed by
 * pf16_maxpool_fwd_argmax on its y.  The workspace is phase 0's
 * (pf16_bn_workspace_size).  Errors as pf16_bn_fwd_bwd; PF16_ERR_ARG when
 * t->y is set; PF16_ERR_UNSUPPORTED for other flags or when 5 rows of w * c
 * values exceed 200 KB; argmax 8-byte aligned. */
int pf16_bn_relu_maxpool_fwd(const pf16_bn_desc* d, const pf16_bn_tensors* t, uint16_t* pooled,
                             uint8_t* argmax, void* ws, size_t ws_bytes, void* stream);

/* ------------------------------------------------- rest of the train step
 * The remaining ops of the ResNet-50 training step (Sec. 5.1), all FP16. */

/* 3x3 max pooling, stride 2, padding 1 (padding never wins), NHWC. */
int pf16_maxpool_fwd(const uint16_t* x, uint16_t* y, int32_t n, int32_t h, int32_t w, int32_t c,
                     void* stream);
/* Backward: each window's gradient goes to the first cell (scan r then s)
 * holding the window maximum; a cell's contributions are added in FP16 in
 * window order.  Writes every element of dx. */
int pf16_maxpool_bwd(const uint16_t* x, const uint16_t* dy, uint16_t* dx, int32_t n, int32_t h,
                     int32_t w, int32_t c, void* stream);
/* The same pair with the window maxima's positions kept between them (a
 * storage choice of this library, no counterpart in the paper): the forward
 * also writes argmax[n][p][q][c] = r*3+s, the position of the first maximum
 * of each window (one byte per output element, 8-byte aligned); the backward
 * reads it instead of x (dx identical to pf16_maxpool_bwd's, bit for bit)
 * and gathers instead of re-scanning the windows.  n, h, w, c are the
 * input's dimensions in both. */
int pf16_maxpool_fwd_argmax(const uint16_t* x, uint16_t* y, uint8_t* argmax, int32_t n, int32_t h,
                            int32_t w, int32_t c, void* stream);
int pf16_maxpool_bwd_argmax(const uint8_t* argmax, const uint16_t* dy, uint16_t* dx, int32_t n,
                            int32_t h, int32_t w, int32_t c, void* stream);
/* Global average pooling: y[n][c] = mean over hw pixels (halving tree). */
int pf16_avgpool_fwd(const uint16_t* x, uint16_t* y, int32_t n, int32_t hw, int32_t c,
                     void* stream);
/* Backward: dx[n][i][c] = rn(dy[n][c] * rn(1/hw)). */
int pf16_avgpool_bwd(const uint16_t* dy, uint16_t* dx, int32_t n, int32_t hw, int32_t c,
                     void* stream);

/* Softmax cross-entropy on logits[b][k] + bias[k] (bias may be NULL) with
 * int32 labels[b] in [0, k): loss (one binary16 scalar, mean over the batch),
 * dlogits[b][k] = (softmax - onehot) / b and dbias[k] = sum_b dlogits (if
 * non-NULL).  k <= 4096; the workspace holds per-row losses. */
size_t pf16_softmax_xent_workspace_size(int32_t b, int32_t k);
int pf16_softmax_xent(const uint16_t* logits, const uint16_t* bias, const int32_t* labels,
                      int32_t b, int32_t k, uint16_t* loss, uint16_t* dlogits, uint16_t* dbias,
                      void* ws, size_t ws_bytes, void* stream);

/* --------------------------------------------------------------- status
 * Waits for `stream`, then returns and clears the device status word of the
 * current device: PF16_OK, PF16_ERR_TIMEOUT after a bounded wait ran out, or
 * PF16_ERR_CUDA if the stream itself reports an error. */
int pf16_sync_status(void* stream);
/* Static, human-readable text for a status code. */
const char* pf16_status_string(int status);
/* Compute capability major*10+minor of the current device, or a negative
 * status if no device is usable.  The kernels need 103 (sm_103a). */
int pf16_device_arch(void);
/* Number of kernels this library has enqueued in this process so far, over
 * all streams and devices; a launch recorded into a CUDA graph during stream
 * capture counts once, when it is recorded.  Monotonic; never fails.  A
 * diagnostic for callers that account for kernel launches (no counterpart in
 * the paper). */
uint64_t pf16_kernel_launches(void);

/* Stream-ordered bounded wait on a device flag: enqueues one single-thread
 * kernel that polls the 32-bit word *flag (device memory, or mapped pinned
 * host memory; acquire loads at system scope) until it equals `value`, for at
 * most timeout_ns nanoseconds of GPU global-timer time.  If the time runs out
 * the kernel records PF16_ERR_TIMEOUT in the device status word (read and
 * cleared by pf16_sync_status) and returns: work queued after it on the
 * stream still runs and the CUDA context stays usable.  This is the failure
 * detection of the library's bounded device-side waits in its smallest form:
 * a producer that never signals (a host thread, a copy on another stream, a
 * peer rank that died) turns into a status code instead of a hung GPU.  No
 * counterpart in the paper.  flag non-NULL (PF16_ERR_NULL) and 4-byte
 * aligned (PF16_ERR_ALIGN); timeout_ns <= 10^10, i.e. 10 s (PF16_ERR_ARG).
 * The flag must be set by something that does not wait on this stream: a
 * kernel that sets it queued behind this one on the same stream never runs
 * in time. */
int pf16_wait_flag(const uint32_t* flag, uint32_t value, uint64_t timeout_ns, void* stream);

/* ------------------------------------------------------------ diagnostics
 * Tensor-core rate probe: the 16-bit dense rate of the instruction the
 * convolutions issue, measured by the library's own MMA-only kernel (the
 * conv rooflines are quoted against a cuBLAS bf16 GEMM; this is the check
 * that FP16 accumulation runs at that rate; not part of the paper's method).
 * One CTA per SM issues reps x 4 tcgen05.mma kind::f16 (M = 128, N = n,
 * K = 16; f16 operands resident in shared memory; f16 accumulator, or f32
 * with f32_accum = 1) into one TMEM accumulator (chains = 1: each MMA adds
 * onto the previous one, as along a GEMM's K loop) or two in turn
 * (chains = 2).  After a warm-up launch, times one launch with CUDA events on
 * `stream` and writes 2*128*n*16 flop per MMA / time, in TFLOP/s, to *tflops.
 * Synchronous (waits for the stream).  n in {64, 128, 192, 256}, f32_accum
 * and chains as above, 1 <= reps <= 2^20 (PF16_ERR_ARG otherwise); tflops
 * non-NULL.  A bounded wait that expires is reported by pf16_sync_status. */
int pf16_tc_rate(int32_t n, int32_t f32_accum, int32_t chains, int32_t reps, double* tflops, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* PF16_H */
