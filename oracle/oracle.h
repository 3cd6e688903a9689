/*
 * ORACLE -- test infrastructure only (see orc_fp16.c).  This header belongs to
 * the oracle alone; the CUDA library never includes it.
 *
 * Tensors are binary16 bit patterns (uint16_t): activations NHWC, conv
 * weights KRSC, all dense.  Results are binary64 unless a function is the
 * bit-exact emulation of an FP16 op sequence.
 */
#ifndef PF16_ORACLE_H
#define PF16_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* binary16 codec and single ops (roundTiesToEven) */
double orc_f16_to_f64(uint16_t h);
uint16_t orc_f64_to_f16(double x);
const double* orc_f16_lut(void);
void orc_f16_decode(const uint16_t* h, double* out, int64_t n);
void orc_f16_encode(const double* x, uint16_t* out, int64_t n);
uint16_t orc_h_add(uint16_t a, uint16_t b);
uint16_t orc_h_sub(uint16_t a, uint16_t b);
uint16_t orc_h_mul(uint16_t a, uint16_t b);

int orc_num_threads(void);

/* Convolutions (dilation 1, groups 1, square stride / pad).
 * For each requested output: V = exact-ish fp64 sum of the products,
 * A = sum of |products|, T = number of (in-range) product terms.
 * idx == NULL means every output in row-major order; otherwise `count`
 * flat output indices.  T may be NULL. */
void orc_conv_fwd(const uint16_t* x, const uint16_t* w, int N, int H, int W, int C, int K, int R,
                  int S, int stride, int pad, const int64_t* idx, int64_t count, double* V,
                  double* A, int32_t* T);
void orc_conv_dgrad(const uint16_t* dy, const uint16_t* w, int N, int H, int W, int C, int K, int R,
                    int S, int stride, int pad, const int64_t* idx, int64_t count, double* V,
                    double* A, int32_t* T);
void orc_conv_wgrad(const uint16_t* x, const uint16_t* dy, int N, int H, int W, int C, int K, int R,
                    int S, int stride, int pad, const int64_t* idx, int64_t count, double* V,
                    double* A, int32_t* T);

/* FP16 SGD with momentum, no master copy: bit-exact emulation, in place. */
void orc_sgd_update(uint16_t* w, uint16_t* v, const uint16_t* g, int64_t n, uint16_t lr,
                    uint16_t momentum, uint16_t wd);

/* Data-parallel gradient average: per element, a pairwise tree of binary16
 * additions over the world's planes in rank order (+0 leaves up to a power of
 * two), then one multiplication by scale (skipped when scale is 1).  Bit-exact. */
void orc_allreduce_combine(const uint16_t* planes, int world, int64_t n, int64_t plane_stride,
                           uint16_t scale, uint16_t* out);

/* BatchNorm over R rows of C channels (training mode, batch statistics). */
void orc_bn_fwd(const uint16_t* x, const uint16_t* gamma, const uint16_t* beta,
                const uint16_t* residual, int64_t R, int C, double eps, double s, int relu,
                double* y, double* mean, double* var, double* invstd);
void orc_bn_bwd(const uint16_t* x, const uint16_t* gamma, const uint16_t* dy,
                const uint16_t* y_saved, int64_t R, int C, double eps, double s, int relu,
                double* dx, double* dgamma, double* dbeta, double* dres);

/* The "swap" variant of a residual block's last BatchNorm (Sec. 4.1: the
 * residual connection and gamma change places): y = gamma * (s * xhat + r) +
 * beta, then optional ReLU; r is the residual input (required). */
void orc_bn_fwd_swap(const uint16_t* x, const uint16_t* gamma, const uint16_t* beta,
                     const uint16_t* residual, int64_t R, int C, double eps, double s, int relu,
                     double* y, double* mean, double* var, double* invstd);
void orc_bn_bwd_swap(const uint16_t* x, const uint16_t* gamma, const uint16_t* dy,
                     const uint16_t* y_saved, const uint16_t* residual, int64_t R, int C, double eps,
                     double s, int relu, double* dx, double* dgamma, double* dbeta, double* dres);

/* 3x3 stride-2 pad-1 max pooling (padding never wins) and its backward. */
void orc_maxpool_fwd(const uint16_t* x, int N, int H, int W, int C, double* y);
void orc_maxpool_bwd(const uint16_t* x, const uint16_t* dy, int N, int H, int W, int C, double* dx,
                     double* A);
/* Global average pooling over H*W and its backward. */
void orc_avgpool_fwd(const uint16_t* x, int N, int HW, int C, double* y);
void orc_avgpool_bwd(const uint16_t* dy, int N, int HW, int C, double* dx);
/* Softmax cross-entropy over logits + bias; mean loss over the batch. */
void orc_softmax_xent(const uint16_t* logits, const uint16_t* bias, const int32_t* labels, int B,
                      int K, double* loss, double* dlogits, double* dbias);

#ifdef __cplusplus
}
#endif
#endif
