/*
 * ORACLE -- test infrastructure only.  Nothing on the product path may link,
 * load or call this code; only tests/, __graft_entry__.smoke() and bench.py's
 * CPU-baseline leg do.
 *
 * Plain, slow, direct-loop definitions of what the pure-FP16 training step
 * computes, evaluated in binary64 on binary16 inputs.  No blocking, no
 * reordering beyond the definitions below; OpenMP only splits independent
 * outputs across threads.
 *
 *  - Convolutions (ResNet-50's layers, paper Sec. 5.1; all arithmetic and
 *    storage FP16, Sec. 5.2): the plain definition of the forward pass and of
 *    its two gradients, returned exactly (binary64 products of binary16
 *    values are exact) with the sum of |terms| for the error bound.
 *  - SGD with momentum and coupled weight decay (the PyTorch ImageNet recipe
 *    the paper adopts, Sec. 5.1) in pure FP16 with no master copy (Sec. 5.2):
 *    each op one binary16 rounding, bit-exact.
 *  - The FP16 gradient average of data-parallel training (Sec. 5.1, 5.2) in a
 *    fixed summation order, bit-exact.
 *  - BatchNorm with batch statistics (Eq. 1, Eq. 2) followed by the x0.25
 *    output scaling inside residual blocks (Sec. 4.2), residual add and ReLU.
 *  - Max pooling, global average pooling and softmax cross-entropy, the rest
 *    of the ResNet-50 training step (Sec. 5.1).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#include "oracle.h"

int orc_num_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

static int out_size(int in, int k, int stride, int pad) { return (in + 2 * pad - k) / stride + 1; }

/* y[n,p,q,k] = sum_{r,s,c} x[n, p*st+r-pad, q*st+s-pad, c] * w[k,r,s,c]  (zero outside x) */
void orc_conv_fwd(const uint16_t* x, const uint16_t* w, int N, int H, int W, int C, int K, int R,
                  int S, int stride, int pad, const int64_t* idx, int64_t count, double* V,
                  double* A, int32_t* T) {
  const double* lut = orc_f16_lut();
  const int P = out_size(H, R, stride, pad), Q = out_size(W, S, stride, pad);
  const int64_t total = (int64_t)N * P * Q * K;
  const int64_t cnt = idx ? count : total;
#pragma omp parallel for schedule(dynamic, 256)
  for (int64_t t = 0; t < cnt; ++t) {
    const int64_t o = idx ? idx[t] : t;
    const int k = (int)(o % K);
    int64_t rest = o / K;
    const int q = (int)(rest % Q);
    rest /= Q;
    const int p = (int)(rest % P);
    const int n = (int)(rest / P);
    double v = 0.0, a = 0.0;
    int nt = 0;
    for (int r = 0; r < R; ++r) {
      const int h = p * stride + r - pad;
      if (h < 0 || h >= H) continue;
      for (int s = 0; s < S; ++s) {
        const int ww = q * stride + s - pad;
        if (ww < 0 || ww >= W) continue;
        const uint16_t* xp = x + (((int64_t)n * H + h) * W + ww) * C;
        const uint16_t* wp = w + (((int64_t)k * R + r) * S + s) * C;
        for (int c = 0; c < C; ++c) {
          const double prod = lut[xp[c]] * lut[wp[c]];
          v += prod;
          a += fabs(prod);
        }
        nt += C;
      }
    }
    V[t] = v;
    A[t] = a;
    if (T) T[t] = nt;
  }
}

/* dx[n,h,w,c] = sum over (k,r,s) with h+pad-r = p*st, w+pad-s = q*st, (p,q) in
   range, of dy[n,p,q,k] * w[k,r,s,c]: the adjoint of orc_conv_fwd in x. */
void orc_conv_dgrad(const uint16_t* dy, const uint16_t* w, int N, int H, int W, int C, int K, int R,
                    int S, int stride, int pad, const int64_t* idx, int64_t count, double* V,
                    double* A, int32_t* T) {
  const double* lut = orc_f16_lut();
  const int P = out_size(H, R, stride, pad), Q = out_size(W, S, stride, pad);
  const int64_t total = (int64_t)N * H * W * C;
  const int64_t cnt = idx ? count : total;
#pragma omp parallel for schedule(dynamic, 256)
  for (int64_t t = 0; t < cnt; ++t) {
    const int64_t o = idx ? idx[t] : t;
    const int c = (int)(o % C);
    int64_t rest = o / C;
    const int ww = (int)(rest % W);
    rest /= W;
    const int h = (int)(rest % H);
    const int n = (int)(rest / H);
    double v = 0.0, a = 0.0;
    int nt = 0;
    for (int r = 0; r < R; ++r) {
      const int hp = h + pad - r;
      if (hp < 0 || hp % stride != 0) continue;
      const int p = hp / stride;
      if (p >= P) continue;
      for (int s = 0; s < S; ++s) {
        const int wq = ww + pad - s;
        if (wq < 0 || wq % stride != 0) continue;
        const int q = wq / stride;
        if (q >= Q) continue;
        const uint16_t* dyp = dy + (((int64_t)n * P + p) * Q + q) * K;
        for (int k = 0; k < K; ++k) {
          const double prod = lut[dyp[k]] * lut[w[(((int64_t)k * R + r) * S + s) * C + c]];
          v += prod;
          a += fabs(prod);
        }
        nt += K;
      }
    }
    V[t] = v;
    A[t] = a;
    if (T) T[t] = nt;
  }
}

/* dw[k,r,s,c] = sum_{n,p,q} dy[n,p,q,k] * x[n, p*st+r-pad, q*st+s-pad, c]:
   the adjoint of orc_conv_fwd in w. */
void orc_conv_wgrad(const uint16_t* x, const uint16_t* dy, int N, int H, int W, int C, int K, int R,
                    int S, int stride, int pad, const int64_t* idx, int64_t count, double* V,
                    double* A, int32_t* T) {
  const double* lut = orc_f16_lut();
  const int P = out_size(H, R, stride, pad), Q = out_size(W, S, stride, pad);
  const int64_t total = (int64_t)K * R * S * C;
  const int64_t cnt = idx ? count : total;
#pragma omp parallel for schedule(dynamic, 16)
  for (int64_t t = 0; t < cnt; ++t) {
    const int64_t o = idx ? idx[t] : t;
    const int c = (int)(o % C);
    int64_t rest = o / C;
    const int s = (int)(rest % S);
    rest /= S;
    const int r = (int)(rest % R);
    const int k = (int)(rest / R);
    double v = 0.0, a = 0.0;
    int nt = 0;
    for (int n = 0; n < N; ++n)
      for (int p = 0; p < P; ++p) {
        const int h = p * stride + r - pad;
        if (h < 0 || h >= H) continue;
        for (int q = 0; q < Q; ++q) {
          const int ww = q * stride + s - pad;
          if (ww < 0 || ww >= W) continue;
          const double prod = lut[dy[(((int64_t)n * P + p) * Q + q) * K + k]] *
                              lut[x[(((int64_t)n * H + h) * W + ww) * C + c]];
          v += prod;
          a += fabs(prod);
          ++nt;
        }
      }
    V[t] = v;
    A[t] = a;
    if (T) T[t] = nt;
  }
}

/* Pure-FP16 SGD step, one binary16 rounding per op, no fused multiply-add:
 *   g' = g + wd*w        (skipped when wd is +0: no decay, e.g. BN parameters)
 *   v' = momentum*v + g'
 *   w' = w - lr*v'
 * The momentum buffer starts at +0; there is no first-step special case. */
void orc_sgd_update(uint16_t* w, uint16_t* v, const uint16_t* g, int64_t n, uint16_t lr,
                    uint16_t momentum, uint16_t wd) {
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) {
    uint16_t gi = g[i];
    if (wd != 0x0000) gi = orc_h_add(gi, orc_h_mul(wd, w[i]));
    const uint16_t vi = orc_h_add(orc_h_mul(momentum, v[i]), gi);
    w[i] = orc_h_sub(w[i], orc_h_mul(lr, vi));
    v[i] = vi;
  }
}

/* The combining step of data-parallel training's gradient exchange (Sec. 5.1:
 * each of `world` GPUs computes the gradient of its own batch; they are
 * averaged before the SGD step, in FP16 like everything else, Sec. 5.2).
 * The reading taken here: the world's gradients are summed first, by a
 * pairwise tree over the ranks in rank order -- at each level, neighbours
 * (0,1), (2,3), ... are added, one binary16 rounding per addition, the rank
 * count padded with +0 leaves up to a power of two -- and the sum is then
 * multiplied by `scale` (normally rn(1/world)), unless scale is 1.  Out of
 * place or in place on plane 0. */
void orc_allreduce_combine(const uint16_t* planes, int world, int64_t n, int64_t plane_stride,
                           uint16_t scale, uint16_t* out) {
  int leaves = 1;
  while (leaves < world) leaves *= 2;
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) {
    uint16_t* t = (uint16_t*)malloc(sizeof(uint16_t) * (size_t)leaves);
    for (int r = 0; r < leaves; ++r) t[r] = r < world ? planes[(int64_t)r * plane_stride + i] : 0x0000;
    for (int width = leaves; width > 1; width /= 2)
      for (int k = 0; k < width / 2; ++k) t[k] = orc_h_add(t[2 * k], t[2 * k + 1]);
    out[i] = scale == 0x3C00 ? t[0] : orc_h_mul(t[0], scale);
    free(t);
  }
}

/* BatchNorm forward, batch statistics over the R rows of each channel:
 *   mean = (1/R) sum x,  var = (1/R) sum (x - mean)^2            (biased)
 *   xhat = (x - mean) / sqrt(var + eps)                          (Eq. 1)
 *   z    = s * (gamma * xhat + beta)                             (Eq. 2, then
 *          the x0.25 scaling of Sec. 4.2; s = 1 for the stem)
 *   y    = relu(z + residual)  (residual and relu optional) */
void orc_bn_fwd(const uint16_t* x, const uint16_t* gamma, const uint16_t* beta,
                const uint16_t* residual, int64_t R, int C, double eps, double s, int relu,
                double* y, double* mean, double* var, double* invstd) {
  const double* lut = orc_f16_lut();
#pragma omp parallel for schedule(dynamic, 1)
  for (int c = 0; c < C; ++c) {
    double sum = 0.0;
    for (int64_t r = 0; r < R; ++r) sum += lut[x[r * C + c]];
    const double mu = sum / (double)R;
    double sq = 0.0;
    for (int64_t r = 0; r < R; ++r) {
      const double d = lut[x[r * C + c]] - mu;
      sq += d * d;
    }
    const double va = sq / (double)R;
    const double is = 1.0 / sqrt(va + eps);
    mean[c] = mu;
    var[c] = va;
    invstd[c] = is;
    const double g = lut[gamma[c]], b = lut[beta[c]];
    for (int64_t r = 0; r < R; ++r) {
      const double xh = (lut[x[r * C + c]] - mu) * is;
      double z = s * (g * xh + b);
      if (residual) z += lut[residual[r * C + c]];
      if (relu && !(z > 0.0)) z = 0.0;
      y[r * C + c] = z;
    }
  }
}

/* BatchNorm backward for the forward above.  dy is the gradient w.r.t. the
 * block output y; the ReLU mask is taken from the saved forward output
 * (y_saved > 0), so both sides decide it on the same binary16 values.
 *   dy'    = dy * [y_saved > 0]        (dy' = dy without relu)
 *   dres   = dy'                       (gradient of the residual input)
 *   dbeta  = s * sum dy',   dgamma = s * sum dy' * xhat
 *   dx     = s*gamma*invstd * (dy' - mean(dy') - xhat * mean(dy' * xhat)) */
void orc_bn_bwd(const uint16_t* x, const uint16_t* gamma, const uint16_t* dy,
                const uint16_t* y_saved, int64_t R, int C, double eps, double s, int relu,
                double* dx, double* dgamma, double* dbeta, double* dres) {
  const double* lut = orc_f16_lut();
#pragma omp parallel for schedule(dynamic, 1)
  for (int c = 0; c < C; ++c) {
    double sum = 0.0;
    for (int64_t r = 0; r < R; ++r) sum += lut[x[r * C + c]];
    const double mu = sum / (double)R;
    double sq = 0.0;
    for (int64_t r = 0; r < R; ++r) {
      const double d = lut[x[r * C + c]] - mu;
      sq += d * d;
    }
    const double is = 1.0 / sqrt(sq / (double)R + eps);
    double s1 = 0.0, s2 = 0.0;
    for (int64_t r = 0; r < R; ++r) {
      double d = lut[dy[r * C + c]];
      if (relu && !(lut[y_saved[r * C + c]] > 0.0)) d = 0.0;
      const double xh = (lut[x[r * C + c]] - mu) * is;
      s1 += d;
      s2 += d * xh;
    }
    dbeta[c] = s * s1;
    dgamma[c] = s * s2;
    const double g = lut[gamma[c]];
    const double m1 = s1 / (double)R, m2 = s2 / (double)R;
    for (int64_t r = 0; r < R; ++r) {
      double d = lut[dy[r * C + c]];
      if (relu && !(lut[y_saved[r * C + c]] > 0.0)) d = 0.0;
      const double xh = (lut[x[r * C + c]] - mu) * is;
      dx[r * C + c] = s * g * is * (d - m1 - xh * m2);
      if (dres) dres[r * C + c] = d;
    }
  }
}

/* BatchNorm "swap" (Sec. 4.1: the residual connection and gamma swap places
 * in a block's last BatchNorm), read as
 *   u = s * xhat + r,   z = gamma * u + beta,   y = relu ? max(z, 0) : z
 * with the same batch statistics of x as orc_bn_fwd. */
void orc_bn_fwd_swap(const uint16_t* x, const uint16_t* gamma, const uint16_t* beta,
                     const uint16_t* residual, int64_t R, int C, double eps, double s, int relu,
                     double* y, double* mean, double* var, double* invstd) {
  const double* lut = orc_f16_lut();
#pragma omp parallel for schedule(dynamic, 1)
  for (int c = 0; c < C; ++c) {
    double sum = 0.0;
    for (int64_t r = 0; r < R; ++r) sum += lut[x[r * C + c]];
    const double mu = sum / (double)R;
    double sq = 0.0;
    for (int64_t r = 0; r < R; ++r) {
      const double d = lut[x[r * C + c]] - mu;
      sq += d * d;
    }
    const double va = sq / (double)R;
    const double is = 1.0 / sqrt(va + eps);
    mean[c] = mu;
    var[c] = va;
    invstd[c] = is;
    const double g = lut[gamma[c]], b = lut[beta[c]];
    for (int64_t r = 0; r < R; ++r) {
      const double xh = (lut[x[r * C + c]] - mu) * is;
      double z = g * (s * xh + lut[residual[r * C + c]]) + b;
      if (relu && !(z > 0.0)) z = 0.0;
      y[r * C + c] = z;
    }
  }
}

/* Its backward, by the chain rule through u and z:
 *   dz     = dy * [y_saved > 0]          (dz = dy without relu)
 *   dbeta  = sum dz,   dgamma = sum dz * u = s * sum dz * xhat + sum dz * r
 *   dres   = gamma * dz                  (gradient of the residual input)
 *   dx     = s*gamma*invstd * (dz - mean(dz) - xhat * mean(dz * xhat)) */
void orc_bn_bwd_swap(const uint16_t* x, const uint16_t* gamma, const uint16_t* dy,
                     const uint16_t* y_saved, const uint16_t* residual, int64_t R, int C, double eps,
                     double s, int relu, double* dx, double* dgamma, double* dbeta, double* dres) {
  const double* lut = orc_f16_lut();
#pragma omp parallel for schedule(dynamic, 1)
  for (int c = 0; c < C; ++c) {
    double sum = 0.0;
    for (int64_t r = 0; r < R; ++r) sum += lut[x[r * C + c]];
    const double mu = sum / (double)R;
    double sq = 0.0;
    for (int64_t r = 0; r < R; ++r) {
      const double d = lut[x[r * C + c]] - mu;
      sq += d * d;
    }
    const double is = 1.0 / sqrt(sq / (double)R + eps);
    double s1 = 0.0, s2 = 0.0, s3 = 0.0;
    for (int64_t r = 0; r < R; ++r) {
      double d = lut[dy[r * C + c]];
      if (relu && !(lut[y_saved[r * C + c]] > 0.0)) d = 0.0;
      const double xh = (lut[x[r * C + c]] - mu) * is;
      s1 += d;
      s2 += d * xh;
      s3 += d * lut[residual[r * C + c]];
    }
    const double g = lut[gamma[c]];
    dbeta[c] = s1;
    dgamma[c] = s * s2 + s3;
    const double m1 = s1 / (double)R, m2 = s2 / (double)R;
    for (int64_t r = 0; r < R; ++r) {
      double d = lut[dy[r * C + c]];
      if (relu && !(lut[y_saved[r * C + c]] > 0.0)) d = 0.0;
      const double xh = (lut[x[r * C + c]] - mu) * is;
      dx[r * C + c] = s * g * is * (d - m1 - xh * m2);
      if (dres) dres[r * C + c] = g * d;
    }
  }
}

/* Max pooling, 3x3 window, stride 2, padding 1 (padded cells never win). */
void orc_maxpool_fwd(const uint16_t* x, int N, int H, int W, int C, double* y) {
  const double* lut = orc_f16_lut();
  const int P = out_size(H, 3, 2, 1), Q = out_size(W, 3, 2, 1);
#pragma omp parallel for schedule(static)
  for (int64_t o = 0; o < (int64_t)N * P * Q; ++o) {
    const int q = (int)(o % Q), p = (int)((o / Q) % P), n = (int)(o / ((int64_t)P * Q));
    for (int c = 0; c < C; ++c) {
      double m = -INFINITY;
      for (int r = 0; r < 3; ++r)
        for (int s = 0; s < 3; ++s) {
          const int h = 2 * p + r - 1, w = 2 * q + s - 1;
          if (h < 0 || h >= H || w < 0 || w >= W) continue;
          const double v = lut[x[(((int64_t)n * H + h) * W + w) * C + c]];
          if (v > m) m = v;
        }
      y[o * C + c] = m;
    }
  }
}

/* Backward: each window's gradient goes to the first cell (row-major scan
   over r then s) that holds the window maximum. */
void orc_maxpool_bwd(const uint16_t* x, const uint16_t* dy, int N, int H, int W, int C, double* dx,
                     double* A) {
  const double* lut = orc_f16_lut();
  const int P = out_size(H, 3, 2, 1), Q = out_size(W, 3, 2, 1);
  memset(dx, 0, sizeof(double) * (size_t)N * H * W * C);
  memset(A, 0, sizeof(double) * (size_t)N * H * W * C);
#pragma omp parallel for schedule(static)
  for (int n = 0; n < N; ++n)
    for (int p = 0; p < P; ++p)
      for (int q = 0; q < Q; ++q)
        for (int c = 0; c < C; ++c) {
          double m = -INFINITY;
          int64_t arg = -1;
          for (int r = 0; r < 3; ++r)
            for (int s = 0; s < 3; ++s) {
              const int h = 2 * p + r - 1, w = 2 * q + s - 1;
              if (h < 0 || h >= H || w < 0 || w >= W) continue;
              const int64_t i = (((int64_t)n * H + h) * W + w) * C + c;
              if (lut[x[i]] > m) {
                m = lut[x[i]];
                arg = i;
              }
            }
          if (arg >= 0) {
            const double g = lut[dy[(((int64_t)n * P + p) * Q + q) * C + c]];
            dx[arg] += g;
            A[arg] += fabs(g);
          }
        }
}

void orc_avgpool_fwd(const uint16_t* x, int N, int HW, int C, double* y) {
  const double* lut = orc_f16_lut();
  for (int n = 0; n < N; ++n)
    for (int c = 0; c < C; ++c) {
      double s = 0.0;
      for (int i = 0; i < HW; ++i) s += lut[x[((int64_t)n * HW + i) * C + c]];
      y[(int64_t)n * C + c] = s / (double)HW;
    }
}

void orc_avgpool_bwd(const uint16_t* dy, int N, int HW, int C, double* dx) {
  const double* lut = orc_f16_lut();
  for (int n = 0; n < N; ++n)
    for (int i = 0; i < HW; ++i)
      for (int c = 0; c < C; ++c)
        dx[((int64_t)n * HW + i) * C + c] = lut[dy[(int64_t)n * C + c]] / (double)HW;
}

/* l = logits + bias; loss_b = logsumexp(l_b) - l_b[label_b]; loss = mean_b;
   dlogits = (softmax(l) - onehot(label)) / B;  dbias = sum_b dlogits. */
void orc_softmax_xent(const uint16_t* logits, const uint16_t* bias, const int32_t* labels, int B,
                      int K, double* loss, double* dlogits, double* dbias) {
  const double* lut = orc_f16_lut();
  double total = 0.0;
  for (int k = 0; k < K; ++k) dbias[k] = 0.0;
  for (int b = 0; b < B; ++b) {
    double m = -INFINITY;
    for (int k = 0; k < K; ++k) {
      const double l = lut[logits[(int64_t)b * K + k]] + (bias ? lut[bias[k]] : 0.0);
      if (l > m) m = l;
    }
    double se = 0.0;
    for (int k = 0; k < K; ++k) {
      const double l = lut[logits[(int64_t)b * K + k]] + (bias ? lut[bias[k]] : 0.0);
      se += exp(l - m);
    }
    const double lse = m + log(se);
    const int lab = labels[b];
    total += lse - (lut[logits[(int64_t)b * K + lab]] + (bias ? lut[bias[lab]] : 0.0));
    for (int k = 0; k < K; ++k) {
      const double l = lut[logits[(int64_t)b * K + k]] + (bias ? lut[bias[k]] : 0.0);
      const double d = (exp(l - lse) - (k == lab ? 1.0 : 0.0)) / (double)B;
      dlogits[(int64_t)b * K + k] = d;
      dbias[k] += d;
    }
  }
  *loss = total / (double)B;
}
