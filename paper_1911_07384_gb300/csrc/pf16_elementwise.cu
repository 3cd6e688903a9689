// Memory-bound kernels of the pure-FP16 ResNet-50 training step: the FP16
// SGD-momentum update, BatchNorm forward/backward with the x0.25 output
// scaling, the split-K FP16 tree reduction of the weight gradient, the stem's
// patch gather, pooling and softmax cross-entropy.  All arithmetic is binary16
// (paper Sec. 5.2), one IEEE rounding per op (add.rn / mul.rn / sub.rn on
// f16x2, never contracted), subnormals kept.  Global traffic is 128-bit.
#include <cuda_fp16.h>

#include "pf16_internal.h"
#include "pf16_ptx.cuh"

namespace pf16 {

namespace {

constexpr uint32_t kHalfHalf2 = 0x38003800u;  // {0.5, 0.5}
constexpr uint32_t kZero2 = 0u;

__host__ __device__ __forceinline__ uint32_t dup2(uint16_t h) { return (uint32_t)h | ((uint32_t)h << 16); }

__device__ __forceinline__ uint4 add4(uint4 a, uint4 b) {
  return make_uint4(hadd2_rn(a.x, b.x), hadd2_rn(a.y, b.y), hadd2_rn(a.z, b.z), hadd2_rn(a.w, b.w));
}
// halving merge: rn(rn(a/2) + rn(b/2)) -- the mean of two nodes, never overflows
__device__ __forceinline__ uint32_t hmerge2(uint32_t a, uint32_t b) {
  return hadd2_rn(hmul2_rn(a, kHalfHalf2), hmul2_rn(b, kHalfHalf2));
}
__device__ __forceinline__ uint4 hmerge4(uint4 a, uint4 b) {
  return make_uint4(hmerge2(a.x, b.x), hmerge2(a.y, b.y), hmerge2(a.z, b.z), hmerge2(a.w, b.w));
}
__device__ __forceinline__ uint4 mul4(uint4 a, uint32_t s) {
  return make_uint4(hmul2_rn(a.x, s), hmul2_rn(a.y, s), hmul2_rn(a.z, s), hmul2_rn(a.w, s));
}
__device__ __forceinline__ uint4 mul4v(uint4 a, uint4 b) {
  return make_uint4(hmul2_rn(a.x, b.x), hmul2_rn(a.y, b.y), hmul2_rn(a.z, b.z), hmul2_rn(a.w, b.w));
}
__device__ __forceinline__ uint4 sub4(uint4 a, uint4 b) {
  return make_uint4(hsub2_rn(a.x, b.x), hsub2_rn(a.y, b.y), hsub2_rn(a.z, b.z), hsub2_rn(a.w, b.w));
}
__device__ __forceinline__ uint4 zero4() { return make_uint4(0, 0, 0, 0); }
__host__ __device__ __forceinline__ int ceil_log2(long long v) {
  int l = 0;
  while ((1ll << l) < v) ++l;
  return l;
}

// x * 2^e for e >= 0 by exact power-of-two steps (each exact unless it overflows)
__device__ __forceinline__ uint4 ldexp4(uint4 v, int e) {
  while (e > 14) {
    v = mul4(v, dup2(0x7400));  // 2^14
    e -= 14;
  }
  const uint16_t pe = (uint16_t)((e + 15) << 10);  // 2^e, 0 <= e <= 14
  return mul4(v, dup2(pe));
}

// positive (> 0, not NaN) test of one binary16 lane, bit-exact
__device__ __forceinline__ bool h_pos(uint32_t h) {
  h &= 0xFFFFu;
  return (h & 0x8000u) == 0 && h != 0 && h <= 0x7C00u;
}
__device__ __forceinline__ uint32_t relu_mask2(uint32_t y) {
  return (h_pos(y) ? 0x0000FFFFu : 0u) | (h_pos(y >> 16) ? 0xFFFF0000u : 0u);
}
__device__ __forceinline__ uint32_t relu2(uint32_t z) { return z & relu_mask2(z); }

// Balanced pairwise tree over a stream of leaves, built as a binary counter:
// after 2^k pushes it holds exactly the perfect tree of those leaves; finish()
// closes the tree as if zero leaves padded the stream to the next power of 2.
template <int MAXL, bool HALVING>
struct Tree4 {
  uint4 st[MAXL];
  unsigned cnt = 0;
  __device__ __forceinline__ static uint4 merge(uint4 a, uint4 b) {
    return HALVING ? hmerge4(a, b) : add4(a, b);
  }
  __device__ __forceinline__ void push(uint4 v) {
#pragma unroll
    for (int l = 0; l < MAXL; ++l) {
      if (cnt & (1u << l)) {
        v = merge(st[l], v);
      } else {
        st[l] = v;
        break;
      }
    }
    ++cnt;
  }
  // Close the tree over 2^levels leaves (cnt <= 2^levels): the pushed leaves
  // followed by zeros.  Walking up from level 0, acc is the rightmost node
  // built so far; a set bit of cnt supplies its left sibling st[l], otherwise
  // its right sibling is an all-zero subtree.
  __device__ __forceinline__ uint4 finish(int levels) {
    uint4 acc = zero4();
    bool have = false;
#pragma unroll
    for (int l = 0; l < MAXL; ++l) {
      if (l < levels) {
        if (cnt & (1u << l)) {
          acc = merge(st[l], have ? acc : zero4());
          have = true;
        } else if (have) {
          acc = merge(acc, zero4());
        }
      } else if (l == levels && (cnt & (1u << l))) {
        acc = st[l];  // cnt == 2^levels: the perfect tree itself
      }
    }
    return acc;
  }
};

}  // namespace

// ============================================================================
// SGD with momentum, pure FP16 (one rounding per op, no FMA):
//   g' = g + wd*w (skipped when wd == +0); v = mom*v + g'; w = w - lr*v
// ============================================================================
__device__ __forceinline__ void sgd2(uint32_t& w, uint32_t& v, uint32_t g, uint32_t lr2,
                                     uint32_t mom2, uint32_t wd2, bool use_wd) {
  if (use_wd) g = hadd2_rn(g, hmul2_rn(wd2, w));
  v = hadd2_rn(hmul2_rn(mom2, v), g);
  w = hsub2_rn(w, hmul2_rn(lr2, v));
}

__global__ void k_sgd(uint16_t* __restrict__ w, uint16_t* __restrict__ v,
                      const uint16_t* __restrict__ g, size_t n, uint32_t lr2, uint32_t mom2,
                      uint32_t wd2, int use_wd) {
  const size_t nvec = n / 8;
  const size_t stride = (size_t)gridDim.x * blockDim.x;
  uint4* W = reinterpret_cast<uint4*>(w);
  uint4* V = reinterpret_cast<uint4*>(v);
  const uint4* G = reinterpret_cast<const uint4*>(g);
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < nvec; i += stride) {
    uint4 a = W[i], b = V[i];
    const uint4 c = __ldg(&G[i]);
    sgd2(a.x, b.x, c.x, lr2, mom2, wd2, use_wd);
    sgd2(a.y, b.y, c.y, lr2, mom2, wd2, use_wd);
    sgd2(a.z, b.z, c.z, lr2, mom2, wd2, use_wd);
    sgd2(a.w, b.w, c.w, lr2, mom2, wd2, use_wd);
    W[i] = a;
    V[i] = b;
  }
  if (blockIdx.x == 0 && threadIdx.x < 8) {  // scalar tail
    const size_t i = nvec * 8 + threadIdx.x;
    if (i < n) {
      uint32_t a = w[i], b = v[i];
      sgd2(a, b, g[i], lr2, mom2, wd2, use_wd);
      w[i] = (uint16_t)a;
      v[i] = (uint16_t)b;
    }
  }
}

cudaError_t launch_sgd(uint16_t* w, uint16_t* v, const uint16_t* g, size_t n, uint16_t lr,
                       uint16_t mom, uint16_t wd, cudaStream_t s) {
  const size_t nvec = n / 8;
  size_t blocks = (nvec + 255) / 256;
  if (blocks < 1) blocks = 1;
  if (blocks > 152 * 16) blocks = 152 * 16;
  k_sgd<<<(unsigned)blocks, 256, 0, s>>>(w, v, g, n, dup2(lr), dup2(mom), dup2(wd), wd != 0);
  return cudaGetLastError();
}

// ============================================================================
// Split-K weight-gradient reduction: out = balanced pairwise FP16 tree over
// the `splits` partial matrices.
// ============================================================================
__global__ void k_splitk_reduce(const uint16_t* __restrict__ parts, int splits, long long rows,
                                int cols, uint16_t* __restrict__ out, long long ldo,
                                int cols_out) {
  const int cpr = cols / 8;
  const long long total = rows * cpr;
  const long long plane = rows * (long long)cols;
  for (long long t = (long long)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (long long)gridDim.x * blockDim.x) {
    const long long r = t / cpr;
    const int cg = (int)(t - r * cpr);
    const uint4* src = reinterpret_cast<const uint4*>(parts + r * cols + cg * 8);
    Tree4<11, false> tree;
    for (int s = 0; s < splits; ++s) tree.push(__ldg(src + (s * plane) / 8));
    const uint4 v = tree.finish(ceil_log2(splits));
    const uint16_t* h = reinterpret_cast<const uint16_t*>(&v);
    uint16_t* o = out + r * ldo + cg * 8;
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (cg * 8 + j < cols_out) o[j] = h[j];
  }
}

cudaError_t launch_splitk_reduce(const uint16_t* parts, int splits, long long rows, int cols,
                                 uint16_t* out, long long ldo, int cols_out, cudaStream_t s) {
  const long long total = rows * (cols / 8);
  long long blocks = (total + 255) / 256;
  if (blocks > 152 * 32) blocks = 152 * 32;
  if (blocks < 1) blocks = 1;
  k_splitk_reduce<<<(unsigned)blocks, 256, 0, s>>>(parts, splits, rows, cols, out, ldo, cols_out);
  return cudaGetLastError();
}

// ============================================================================
// Stem patch gather (c = 3 cannot be fetched by TMA: a pixel is 6 bytes).
// col[m][j], m = (n, p, q), j = (r*S + s)*C + c < R*S*C, zero-padded to kcol.
// ============================================================================
__global__ void k_stem_im2col(const uint16_t* __restrict__ x, uint16_t* __restrict__ col, int N,
                              int H, int W, int P, int Q, int R, int S, int C, int stride, int pad,
                              int kcol) {
  const int groups = kcol / 8;
  const long long total = (long long)N * P * Q * groups;
  const int kin = R * S * C;
  for (long long t = (long long)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (long long)gridDim.x * blockDim.x) {
    const long long m = t / groups;
    const int g = (int)(t - m * groups);
    const int q = (int)(m % Q);
    const int p = (int)((m / Q) % P);
    const int n = (int)(m / ((long long)P * Q));
    uint16_t v[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const int j = g * 8 + e;
      uint16_t val = 0;
      if (j < kin) {
        const int c = j % C, rs = j / C;
        const int s = rs % S, r = rs / S;
        const int h = p * stride + r - pad, w = q * stride + s - pad;
        if (h >= 0 && h < H && w >= 0 && w < W) val = x[(((long long)n * H + h) * W + w) * C + c];
      }
      v[e] = val;
    }
    *reinterpret_cast<uint4*>(col + m * kcol + g * 8) = *reinterpret_cast<uint4*>(v);
  }
}

cudaError_t launch_stem_im2col(const uint16_t* x, uint16_t* col, int N, int H, int W, int P, int Q,
                               int R, int S, int C, int stride, int pad, int kcol,
                               cudaStream_t s) {
  const long long total = (long long)N * P * Q * (kcol / 8);
  long long blocks = (total + 255) / 256;
  if (blocks > 152 * 64) blocks = 152 * 64;
  k_stem_im2col<<<(unsigned)blocks, 256, 0, s>>>(x, col, N, H, W, P, Q, R, S, C, stride, pad, kcol);
  return cudaGetLastError();
}

__global__ void k_pad_rows(const uint16_t* __restrict__ w, uint16_t* __restrict__ wp, int K, int kin,
                           int kcol) {
  const int total = K * kcol;
  for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < total; t += gridDim.x * blockDim.x) {
    const int k = t / kcol, j = t - k * kcol;
    wp[t] = j < kin ? w[k * kin + j] : (uint16_t)0;
  }
}

cudaError_t launch_pad_rows(const uint16_t* w, uint16_t* wp, int K, int kin, int kcol,
                            cudaStream_t s) {
  const int blocks = (K * kcol + 255) / 256;
  k_pad_rows<<<blocks, 256, 0, s>>>(w, wp, K, kin, kcol);
  return cudaGetLastError();
}

cudaError_t launch_fill_zero(uint16_t* p, size_t n, cudaStream_t s) {
  return cudaMemsetAsync(p, 0, n * sizeof(uint16_t), s);
}

// ============================================================================
// BatchNorm (Eq. 1, Eq. 2, then x post_scale, + residual, ReLU), FP16 only.
//
// Statistics are means over the R rows of each channel computed as balanced
// "halving" trees (node = rn(rn(a/2) + rn(b/2))) over R zero-padded to 2^L
// leaves: thread-level trees over rows_per_thread leaves, a shared-memory
// tree over the block's row groups, then a tree over the blocks' results in a
// second kernel, and one final multiplication by rn(2^L / R).  Sums (for
// dgamma, dbeta) are the same tree scaled back by 2^L exactly.
// ============================================================================
namespace {

constexpr int kBnThreads = 256;
constexpr int kBnMaxL = 8;  // rows per thread <= 256

struct BnGeom {
  int tc;   // threads per row (channel groups of 8)
  int rpb;  // row groups per block (power of two)
  int rpt;  // rows per thread (power of two)
};

__host__ __device__ inline BnGeom bn_geom(int C, int rows_per_block) {
  BnGeom g;
  g.tc = C / 8;
  int rpb = 1;
  while (rpb * 2 * g.tc <= kBnThreads) rpb *= 2;
  g.rpb = rpb;
  g.rpt = rows_per_block / rpb;
  return g;
}

enum { BN_STAT_MEAN = 0, BN_STAT_VAR = 1, BN_STAT_BWD = 2 };

// Partial per-block means.  ws_out[block][C] (and ws_out2 for the backward).
template <int MODE>
__global__ void __launch_bounds__(kBnThreads)
    k_bn_partial(const uint16_t* __restrict__ x, const uint16_t* __restrict__ dy,
                 const uint16_t* __restrict__ y_saved, const uint16_t* __restrict__ mean,
                 const uint16_t* __restrict__ invstd, int R, int C, int rows_per_block, int relu,
                 uint16_t* __restrict__ ws_out, uint16_t* __restrict__ ws_out2) {
  extern __shared__ uint4 sh[];
  const BnGeom g = bn_geom(C, rows_per_block);
  const int t = threadIdx.x;
  const bool active = t < g.tc * g.rpb;
  const int cg = t % g.tc, rg = t / g.tc;
  const long long row0 = (long long)blockIdx.x * rows_per_block;
  Tree4<kBnMaxL, true> t1, t2;
  uint4 mu = zero4(), is = zero4();
  if (active && MODE != BN_STAT_MEAN) mu = __ldg(reinterpret_cast<const uint4*>(mean) + cg);
  if (active && MODE == BN_STAT_BWD) is = __ldg(reinterpret_cast<const uint4*>(invstd) + cg);
  if (active) {
    for (int i = 0; i < g.rpt; ++i) {
      const long long r = row0 + rg + (long long)i * g.rpb;
      uint4 l1 = zero4(), l2 = zero4();
      if (r < R) {
        const long long off = (r * C) / 8 + cg;
        const uint4 xv = __ldg(reinterpret_cast<const uint4*>(x) + off);
        if (MODE == BN_STAT_MEAN) {
          l1 = xv;
        } else if (MODE == BN_STAT_VAR) {
          const uint4 d = sub4(xv, mu);
          l1 = mul4v(d, d);
        } else {
          uint4 d = __ldg(reinterpret_cast<const uint4*>(dy) + off);
          if (relu) {
            const uint4 ys = __ldg(reinterpret_cast<const uint4*>(y_saved) + off);
            d.x &= relu_mask2(ys.x);
            d.y &= relu_mask2(ys.y);
            d.z &= relu_mask2(ys.z);
            d.w &= relu_mask2(ys.w);
          }
          const uint4 xh = mul4v(sub4(xv, mu), is);
          l1 = d;
          l2 = mul4v(d, xh);
        }
      }
      t1.push(l1);
      if (MODE == BN_STAT_BWD) t2.push(l2);
    }
  }
  const int lv = 31 - __clz(g.rpt);
  uint4* s1 = sh;
  uint4* s2 = sh + kBnThreads;
  if (active) {
    s1[t] = t1.finish(lv);
    if (MODE == BN_STAT_BWD) s2[t] = t2.finish(lv);
  }
  __syncthreads();
  // tree over row groups: partner rg ^ half
  for (int half = g.rpb / 2; half >= 1; half /= 2) {
    if (active && rg < half) {
      const int o = (rg + half) * g.tc + cg;
      s1[t] = hmerge4(s1[t], s1[o]);
      if (MODE == BN_STAT_BWD) s2[t] = hmerge4(s2[t], s2[o]);
    }
    __syncthreads();
  }
  if (active && rg == 0) {
    reinterpret_cast<uint4*>(ws_out)[(long long)blockIdx.x * g.tc + cg] = s1[t];
    if (MODE == BN_STAT_BWD) reinterpret_cast<uint4*>(ws_out2)[(long long)blockIdx.x * g.tc + cg] = s2[t];
  }
}

// Tree over the per-block results (blocks zero-padded to blocks_pow2).  One
// CTA of 256 threads per channel group of 8.
template <int MODE>
__global__ void __launch_bounds__(256)
    k_bn_final(const uint16_t* __restrict__ ws1, const uint16_t* __restrict__ ws2, int C,
               int blocks, int blocks_pow2, int total_levels, uint16_t ratio, uint16_t eps,
               uint16_t post_scale, const uint16_t* __restrict__ gamma, uint16_t* __restrict__ out1,
               uint16_t* __restrict__ out2, uint16_t* __restrict__ dgamma,
               uint16_t* __restrict__ dbeta, uint16_t* __restrict__ m_out) {
  __shared__ uint4 s1[256], s2[256];
  const int tc = C / 8;
  const int cg = blockIdx.x;
  const int t = threadIdx.x;
  const int nthr = blocks_pow2 < 256 ? blocks_pow2 : 256;
  const int per = blocks_pow2 / nthr;  // power of two
  if (t < nthr) {
    Tree4<12, true> a, b;
    for (int i = 0; i < per; ++i) {
      const int blk = t * per + i;
      uint4 v1 = zero4(), v2 = zero4();
      if (blk < blocks) {
        v1 = __ldg(reinterpret_cast<const uint4*>(ws1) + (long long)blk * tc + cg);
        if (MODE == BN_STAT_BWD) v2 = __ldg(reinterpret_cast<const uint4*>(ws2) + (long long)blk * tc + cg);
      }
      a.push(v1);
      if (MODE == BN_STAT_BWD) b.push(v2);
    }
    const int lv = 31 - __clz(per);
    s1[t] = a.finish(lv);
    if (MODE == BN_STAT_BWD) s2[t] = b.finish(lv);
  }
  __syncthreads();
  for (int half = nthr / 2; half >= 1; half /= 2) {
    if (t < half) {
      s1[t] = hmerge4(s1[t], s1[t + half]);
      if (MODE == BN_STAT_BWD) s2[t] = hmerge4(s2[t], s2[t + half]);
    }
    __syncthreads();
  }
  if (t != 0) return;
  const uint32_t ratio2 = dup2(ratio);
  if (MODE == BN_STAT_MEAN) {
    reinterpret_cast<uint4*>(out1)[cg] = mul4(s1[0], ratio2);
  } else if (MODE == BN_STAT_VAR) {
    const uint4 var = mul4(s1[0], ratio2);
    const uint4 ve = add4(var, make_uint4(dup2(eps), dup2(eps), dup2(eps), dup2(eps)));
    uint4 r;
    const __half2* hv = reinterpret_cast<const __half2*>(&ve);
    __half2* hr = reinterpret_cast<__half2*>(&r);
#pragma unroll
    for (int j = 0; j < 4; ++j) hr[j] = h2rsqrt(hv[j]);
    reinterpret_cast<uint4*>(out2)[cg] = r;
  } else {
    // means for the elementwise pass, and the sums (tree * 2^L) for dbeta / dgamma
    const uint4 m1 = mul4(s1[0], ratio2), m2 = mul4(s2[0], ratio2);
    reinterpret_cast<uint4*>(m_out)[cg] = m1;
    reinterpret_cast<uint4*>(m_out)[tc + cg] = m2;
    const uint32_t ps = dup2(post_scale);
    reinterpret_cast<uint4*>(dbeta)[cg] = mul4(ldexp4(s1[0], total_levels), ps);
    reinterpret_cast<uint4*>(dgamma)[cg] = mul4(ldexp4(s2[0], total_levels), ps);
  }
}

__global__ void __launch_bounds__(256)
    k_bn_apply(const uint16_t* __restrict__ x, const uint16_t* __restrict__ gamma,
               const uint16_t* __restrict__ beta, const uint16_t* __restrict__ mean,
               const uint16_t* __restrict__ invstd, const uint16_t* __restrict__ residual,
               uint16_t* __restrict__ y, long long total_vec, int tc, uint16_t post_scale,
               int relu) {
  const uint32_t ps = dup2(post_scale);
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total_vec;
       i += (long long)gridDim.x * blockDim.x) {
    const int cg = (int)(i % tc);
    const uint4 xv = __ldg(reinterpret_cast<const uint4*>(x) + i);
    const uint4 mu = __ldg(reinterpret_cast<const uint4*>(mean) + cg);
    const uint4 is = __ldg(reinterpret_cast<const uint4*>(invstd) + cg);
    const uint4 ga = __ldg(reinterpret_cast<const uint4*>(gamma) + cg);
    const uint4 be = __ldg(reinterpret_cast<const uint4*>(beta) + cg);
    const uint4 xh = mul4v(sub4(xv, mu), is);         // Eq. 1
    uint4 z = mul4(add4(mul4v(ga, xh), be), ps);      // Eq. 2, then x post_scale
    if (residual) z = add4(z, __ldg(reinterpret_cast<const uint4*>(residual) + i));
    if (relu) {
      z.x = relu2(z.x);
      z.y = relu2(z.y);
      z.z = relu2(z.z);
      z.w = relu2(z.w);
    }
    reinterpret_cast<uint4*>(y)[i] = z;
  }
}

__global__ void __launch_bounds__(256)
    k_bn_bwd_apply(const uint16_t* __restrict__ x, const uint16_t* __restrict__ gamma,
                   const uint16_t* __restrict__ mean, const uint16_t* __restrict__ invstd,
                   const uint16_t* __restrict__ dy, const uint16_t* __restrict__ y_saved,
                   const uint16_t* __restrict__ mm, uint16_t* __restrict__ dx,
                   uint16_t* __restrict__ dres, long long total_vec, int tc, uint16_t post_scale,
                   int relu) {
  const uint32_t ps = dup2(post_scale);
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total_vec;
       i += (long long)gridDim.x * blockDim.x) {
    const int cg = (int)(i % tc);
    uint4 d = __ldg(reinterpret_cast<const uint4*>(dy) + i);
    if (relu) {
      const uint4 ys = __ldg(reinterpret_cast<const uint4*>(y_saved) + i);
      d.x &= relu_mask2(ys.x);
      d.y &= relu_mask2(ys.y);
      d.z &= relu_mask2(ys.z);
      d.w &= relu_mask2(ys.w);
    }
    const uint4 xv = __ldg(reinterpret_cast<const uint4*>(x) + i);
    const uint4 mu = __ldg(reinterpret_cast<const uint4*>(mean) + cg);
    const uint4 is = __ldg(reinterpret_cast<const uint4*>(invstd) + cg);
    const uint4 ga = __ldg(reinterpret_cast<const uint4*>(gamma) + cg);
    const uint4 m1 = __ldg(reinterpret_cast<const uint4*>(mm) + cg);
    const uint4 m2 = __ldg(reinterpret_cast<const uint4*>(mm) + tc + cg);
    const uint4 xh = mul4v(sub4(xv, mu), is);
    const uint4 k = mul4v(mul4(ga, ps), is);          // s * gamma * invstd
    const uint4 t = sub4(sub4(d, m1), mul4v(xh, m2));  // dy' - mean(dy') - xhat*mean(dy'*xhat)
    reinterpret_cast<uint4*>(dx)[i] = mul4v(k, t);
    if (dres) reinterpret_cast<uint4*>(dres)[i] = d;
  }
}

unsigned grid_for(long long work, int per_block, int cap) {
  long long b = (work + per_block - 1) / per_block;
  if (b < 1) b = 1;
  if (b > cap) b = cap;
  return (unsigned)b;
}

}  // namespace

void bn_plan(int R, int C, BnLaunch* b) {
  b->R = R;
  b->C = C;
  const BnGeom g0 = bn_geom(C, 1);
  // rows per thread: aim for about 4 CTAs per SM, 8..128 rows per thread
  int rpt = 8;
  while (rpt < 128 && (long long)R / ((long long)g0.rpb * rpt * 2) >= 152 * 4) rpt *= 2;
  b->rows_per_block = g0.rpb * rpt;
  b->blocks = (int)(((long long)R + b->rows_per_block - 1) / b->rows_per_block);
  int p2 = 1;
  while (p2 < b->blocks) p2 *= 2;
  b->blocks_pow2 = p2;
}

size_t bn_ws_bytes(const BnLaunch& b) {
  // two per-block partial planes + the two per-channel means of the backward
  return (size_t)2 * b.blocks * b.C * sizeof(uint16_t) + (size_t)2 * b.C * sizeof(uint16_t) + 256;
}

static uint16_t f16_bits_host(float f) {
  __half h = __float2half_rn(f);
  return *reinterpret_cast<uint16_t*>(&h);
}

static void bn_scale_consts(const BnLaunch& b, uint16_t* ratio, int* levels) {
  const long long leaves = (long long)b.rows_per_block * b.blocks_pow2;
  int L = 0;
  while ((1ll << L) < leaves) ++L;
  *levels = L;
  *ratio = f16_bits_host((float)((double)leaves / (double)b.R));
}

cudaError_t launch_bn_fwd(const BnLaunch& b, const uint16_t* x, const uint16_t* gamma,
                          const uint16_t* beta, const uint16_t* residual, uint16_t* y,
                          uint16_t* mean, uint16_t* invstd, uint16_t* ws, cudaStream_t s) {
  uint16_t ratio;
  int L;
  bn_scale_consts(b, &ratio, &L);
  const size_t shm = 2 * kBnThreads * sizeof(uint4);
  uint16_t* part = ws;
  k_bn_partial<BN_STAT_MEAN><<<b.blocks, kBnThreads, shm, s>>>(x, nullptr, nullptr, nullptr, nullptr,
                                                               b.R, b.C, b.rows_per_block, 0, part,
                                                               nullptr);
  k_bn_final<BN_STAT_MEAN><<<b.C / 8, 256, 0, s>>>(part, nullptr, b.C, b.blocks, b.blocks_pow2, L,
                                                   ratio, b.eps, b.post_scale, gamma, mean, nullptr,
                                                   nullptr, nullptr, nullptr);
  k_bn_partial<BN_STAT_VAR><<<b.blocks, kBnThreads, shm, s>>>(x, nullptr, nullptr, mean, nullptr, b.R,
                                                              b.C, b.rows_per_block, 0, part,
                                                              nullptr);
  k_bn_final<BN_STAT_VAR><<<b.C / 8, 256, 0, s>>>(part, nullptr, b.C, b.blocks, b.blocks_pow2, L,
                                                  ratio, b.eps, b.post_scale, gamma, nullptr, invstd,
                                                  nullptr, nullptr, nullptr);
  const long long tv = (long long)b.R * b.C / 8;
  k_bn_apply<<<grid_for(tv, 256, 152 * 16), 256, 0, s>>>(x, gamma, beta, mean, invstd, residual, y, tv, b.C / 8,
                                                         b.post_scale, b.relu);
  return cudaGetLastError();
}

cudaError_t launch_bn_bwd(const BnLaunch& b, const uint16_t* x, const uint16_t* gamma,
                          const uint16_t* mean, const uint16_t* invstd, const uint16_t* dy,
                          const uint16_t* y_saved, uint16_t* dx, uint16_t* dgamma,
                          uint16_t* dbeta, uint16_t* dres, uint16_t* ws, cudaStream_t s) {
  uint16_t ratio;
  int L;
  bn_scale_consts(b, &ratio, &L);
  const size_t shm = 2 * kBnThreads * sizeof(uint4);
  uint16_t* p1 = ws;
  uint16_t* p2 = ws + (size_t)b.blocks * b.C;
  uint16_t* mm = ws + (size_t)2 * b.blocks * b.C;
  k_bn_partial<BN_STAT_BWD><<<b.blocks, kBnThreads, shm, s>>>(x, dy, y_saved, mean, invstd, b.R, b.C,
                                                              b.rows_per_block, b.relu, p1, p2);
  k_bn_final<BN_STAT_BWD><<<b.C / 8, 256, 0, s>>>(p1, p2, b.C, b.blocks, b.blocks_pow2, L, ratio,
                                                  b.eps, b.post_scale, gamma, nullptr, nullptr,
                                                  dgamma, dbeta, mm);
  const long long tv = (long long)b.R * b.C / 8;
  k_bn_bwd_apply<<<grid_for(tv, 256, 152 * 16), 256, 0, s>>>(x, gamma, mean, invstd, dy, y_saved, mm, dx,
                                                             dres, tv, b.C / 8, b.post_scale, b.relu);
  return cudaGetLastError();
}

// ============================================================================
// Max pooling 3x3 / stride 2 / pad 1 and its backward (first-max rule).
// ============================================================================
__global__ void k_maxpool_fwd(const uint16_t* __restrict__ x, uint16_t* __restrict__ y, int N, int H,
                              int W, int C, int P, int Q) {
  const int tc = C / 8;
  const long long total = (long long)N * P * Q * tc;
  for (long long t = (long long)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (long long)gridDim.x * blockDim.x) {
    const int cg = (int)(t % tc);
    const long long o = t / tc;
    const int q = (int)(o % Q), p = (int)((o / Q) % P), n = (int)(o / ((long long)P * Q));
    float m[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) m[e] = -INFINITY;
    for (int r = 0; r < 3; ++r) {
      const int h = 2 * p + r - 1;
      if (h < 0 || h >= H) continue;
      for (int s = 0; s < 3; ++s) {
        const int w = 2 * q + s - 1;
        if (w < 0 || w >= W) continue;
        const uint4 v = __ldg(reinterpret_cast<const uint4*>(x + (((long long)n * H + h) * W + w) * C) + cg);
        const __half* hv = reinterpret_cast<const __half*>(&v);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float f = __half2float(hv[e]);
          if (f > m[e]) m[e] = f;
        }
      }
    }
    uint4 out;
    __half* ho = reinterpret_cast<__half*>(&out);
#pragma unroll
    for (int e = 0; e < 8; ++e) ho[e] = __float2half_rn(m[e]);  // exact: m is a binary16 value
    reinterpret_cast<uint4*>(y)[t] = out;
  }
}

__global__ void k_maxpool_bwd(const uint16_t* __restrict__ x, const uint16_t* __restrict__ dy,
                              uint16_t* __restrict__ dx, int N, int H, int W, int C, int P, int Q) {
  const int tc = C / 8;
  const long long total = (long long)N * H * W * tc;
  for (long long t = (long long)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (long long)gridDim.x * blockDim.x) {
    const int cg = (int)(t % tc);
    const long long pix = t / tc;
    const int w = (int)(pix % W), h = (int)((pix / W) % H), n = (int)(pix / ((long long)H * W));
    uint32_t acc[4] = {0, 0, 0, 0};
    const int p_lo = h / 2, p_hi = min(P - 1, (h + 1) / 2);
    const int q_lo = w / 2, q_hi = min(Q - 1, (w + 1) / 2);
    for (int p = p_lo; p <= p_hi; ++p) {
      if (h < 2 * p - 1 || h > 2 * p + 1) continue;
      for (int q = q_lo; q <= q_hi; ++q) {
        if (w < 2 * q - 1 || w > 2 * q + 1) continue;
        // argmax of window (p, q): first maximum in r-then-s order
        float m[8];
        int arg[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          m[e] = -INFINITY;
          arg[e] = -1;
        }
        for (int r = 0; r < 3; ++r) {
          const int hh = 2 * p + r - 1;
          if (hh < 0 || hh >= H) continue;
          for (int s = 0; s < 3; ++s) {
            const int ww = 2 * q + s - 1;
            if (ww < 0 || ww >= W) continue;
            const uint4 v =
                __ldg(reinterpret_cast<const uint4*>(x + (((long long)n * H + hh) * W + ww) * C) + cg);
            const __half* hv = reinterpret_cast<const __half*>(&v);
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const float f = __half2float(hv[e]);
              if (f > m[e]) {
                m[e] = f;
                arg[e] = hh * W + ww;
              }
            }
          }
        }
        const uint4 g = __ldg(reinterpret_cast<const uint4*>(dy + (((long long)n * P + p) * Q + q) * C) + cg);
        const uint32_t* gw = reinterpret_cast<const uint32_t*>(&g);
        const int me = h * W + w;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint32_t sel = (arg[2 * j] == me ? 0x0000FFFFu : 0u) | (arg[2 * j + 1] == me ? 0xFFFF0000u : 0u);
          if (sel) acc[j] = hadd2_rn(acc[j], gw[j] & sel);
        }
      }
    }
    reinterpret_cast<uint4*>(dx)[t] = make_uint4(acc[0], acc[1], acc[2], acc[3]);
  }
}

cudaError_t launch_maxpool_fwd(const uint16_t* x, uint16_t* y, int N, int H, int W, int C,
                               cudaStream_t s) {
  const int P = (H - 1) / 2 + 1, Q = (W - 1) / 2 + 1;
  const long long total = (long long)N * P * Q * (C / 8);
  k_maxpool_fwd<<<grid_for(total, 256, 152 * 16), 256, 0, s>>>(x, y, N, H, W, C, P, Q);
  return cudaGetLastError();
}

cudaError_t launch_maxpool_bwd(const uint16_t* x, const uint16_t* dy, uint16_t* dx, int N, int H,
                               int W, int C, cudaStream_t s) {
  const int P = (H - 1) / 2 + 1, Q = (W - 1) / 2 + 1;
  const long long total = (long long)N * H * W * (C / 8);
  k_maxpool_bwd<<<grid_for(total, 256, 152 * 16), 256, 0, s>>>(x, dy, dx, N, H, W, C, P, Q);
  return cudaGetLastError();
}

// ============================================================================
// Global average pooling (halving tree over hw padded to 2^L, x rn(2^L/hw)).
// ============================================================================
__global__ void k_avgpool_fwd(const uint16_t* __restrict__ x, uint16_t* __restrict__ y, int N, int HW,
                              int C, int levels, uint16_t ratio) {
  const int tc = C / 8;
  const long long total = (long long)N * tc;
  for (long long t = (long long)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (long long)gridDim.x * blockDim.x) {
    const int cg = (int)(t % tc);
    const long long n = t / tc;
    Tree4<12, true> tree;
    for (int i = 0; i < HW; ++i)
      tree.push(__ldg(reinterpret_cast<const uint4*>(x + (n * HW + i) * C) + cg));
    reinterpret_cast<uint4*>(y)[t] = mul4(tree.finish(levels), dup2(ratio));
  }
}

__global__ void k_avgpool_bwd(const uint16_t* __restrict__ dy, uint16_t* __restrict__ dx, int N,
                              int HW, int C, uint16_t inv) {
  const int tc = C / 8;
  const long long total = (long long)N * HW * tc;
  for (long long t = (long long)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (long long)gridDim.x * blockDim.x) {
    const int cg = (int)(t % tc);
    const long long n = t / ((long long)HW * tc);
    reinterpret_cast<uint4*>(dx)[t] = mul4(__ldg(reinterpret_cast<const uint4*>(dy + n * C) + cg), dup2(inv));
  }
}

cudaError_t launch_avgpool_fwd(const uint16_t* x, uint16_t* y, int N, int HW, int C,
                               cudaStream_t s) {
  int L = 0;
  while ((1 << L) < HW) ++L;
  const uint16_t ratio = f16_bits_host((float)((double)(1 << L) / HW));
  const long long total = (long long)N * (C / 8);
  k_avgpool_fwd<<<grid_for(total, 128, 152 * 16), 128, 0, s>>>(x, y, N, HW, C, L, ratio);
  return cudaGetLastError();
}

cudaError_t launch_avgpool_bwd(const uint16_t* dy, uint16_t* dx, int N, int HW, int C,
                               cudaStream_t s) {
  const uint16_t inv = f16_bits_host((float)(1.0 / HW));
  const long long total = (long long)N * HW * (C / 8);
  k_avgpool_bwd<<<grid_for(total, 256, 152 * 16), 256, 0, s>>>(dy, dx, N, HW, C, inv);
  return cudaGetLastError();
}

// ============================================================================
// Softmax cross-entropy: per row (one CTA), l = rn(z + b), m = max l,
// S = pairwise FP16 sum of exp(rn(l - m)), lse = rn(m + log S),
// dlogits = rn(rn(exp(rn(l - lse)) - onehot) * rn(1/B)), loss_b = rn(lse - l_label);
// then the batch mean of loss_b (halving tree) and dbias = pairwise column sums.
// ============================================================================
namespace {
constexpr int kSmThreads = 256;

__device__ __forceinline__ __half hb(uint16_t u) { return __ushort_as_half(u); }
__device__ __forceinline__ uint16_t bh(__half h) { return __half_as_ushort(h); }
__device__ __forceinline__ __half hadd(__half a, __half b) { return hb((uint16_t)hadd2_rn(bh(a), bh(b))); }
__device__ __forceinline__ __half hsub(__half a, __half b) { return hb((uint16_t)hsub2_rn(bh(a), bh(b))); }
__device__ __forceinline__ __half hmul(__half a, __half b) { return hb((uint16_t)hmul2_rn(bh(a), bh(b))); }
}  // namespace

__global__ void __launch_bounds__(kSmThreads)
    k_softmax_rows(const uint16_t* __restrict__ logits, const uint16_t* __restrict__ bias,
                   const int32_t* __restrict__ labels, int K, uint16_t invB,
                   uint16_t* __restrict__ dlogits, uint16_t* __restrict__ row_loss) {
  __shared__ float smax[kSmThreads / 32];
  __shared__ uint16_t ssum[kSmThreads];
  __shared__ __half s_lse;
  const int b = blockIdx.x, t = threadIdx.x;
  const uint16_t* z = logits + (long long)b * K;
  // pass 1: max of l
  float mx = -INFINITY;
  for (int k = t; k < K; k += kSmThreads) {
    const __half l = bias ? hadd(hb(z[k]), hb(bias[k])) : hb(z[k]);
    mx = fmaxf(mx, __half2float(l));
  }
#pragma unroll
  for (int o = 16; o >= 1; o /= 2) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  if ((t & 31) == 0) smax[t >> 5] = mx;
  __syncthreads();
  if (t < 32) {
    float v = t < kSmThreads / 32 ? smax[t] : -INFINITY;
#pragma unroll
    for (int o = 16; o >= 1; o /= 2) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    if (t == 0) smax[0] = v;
  }
  __syncthreads();
  const __half m = __float2half_rn(smax[0]);  // exact: the max of binary16 values
  // pass 2: S = sum exp(rn(l - m)) as a pairwise tree (thread trees, then across threads)
  uint16_t st[8];
  unsigned cnt = 0;
  for (int k = t; k < K; k += kSmThreads) {
    const __half l = bias ? hadd(hb(z[k]), hb(bias[k])) : hb(z[k]);
    uint16_t v = bh(hexp(hsub(l, m)));
#pragma unroll
    for (int lv = 0; lv < 8; ++lv) {
      if (cnt & (1u << lv)) {
        v = bh(hadd(hb(st[lv]), hb(v)));
      } else {
        st[lv] = v;
        break;
      }
    }
    ++cnt;
  }
  uint16_t acc = 0;
  bool have = false;
#pragma unroll
  for (int lv = 0; lv < 8; ++lv)
    if (cnt & (1u << lv)) {
      acc = have ? bh(hadd(hb(st[lv]), hb(acc))) : st[lv];
      have = true;
    }
  ssum[t] = acc;
  __syncthreads();
  for (int half = kSmThreads / 2; half >= 1; half /= 2) {
    if (t < half) ssum[t] = bh(hadd(hb(ssum[t]), hb(ssum[t + half])));
    __syncthreads();
  }
  if (t == 0) s_lse = hadd(m, hlog(hb(ssum[0])));
  __syncthreads();
  const __half lse = s_lse;
  const int lab = labels[b];
  for (int k = t; k < K; k += kSmThreads) {
    const __half l = bias ? hadd(hb(z[k]), hb(bias[k])) : hb(z[k]);
    __half p = hexp(hsub(l, lse));
    if (k == lab) {
      p = hsub(p, __float2half_rn(1.0f));
      row_loss[b] = bh(hsub(lse, l));
    }
    dlogits[(long long)b * K + k] = bh(hmul(p, hb(invB)));
  }
}

__global__ void k_softmax_cols(const uint16_t* __restrict__ dlogits, const uint16_t* __restrict__ row_loss,
                               int B, int K, int levels, uint16_t ratio, uint16_t* __restrict__ dbias,
                               uint16_t* __restrict__ loss) {
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (dbias && k < K) {
    uint16_t st[16];
    unsigned cnt = 0;
    for (int b = 0; b < B; ++b) {
      uint16_t v = dlogits[(long long)b * K + k];
#pragma unroll
      for (int lv = 0; lv < 16; ++lv) {
        if (cnt & (1u << lv)) {
          v = bh(hadd(hb(st[lv]), hb(v)));
        } else {
          st[lv] = v;
          break;
        }
      }
      ++cnt;
    }
    uint16_t acc = 0;
    bool have = false;
#pragma unroll
    for (int lv = 0; lv < 16; ++lv)
      if (cnt & (1u << lv)) {
        acc = have ? bh(hadd(hb(st[lv]), hb(acc))) : st[lv];
        have = true;
      }
    dbias[k] = acc;
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    // batch mean of the row losses: halving tree over B padded to 2^levels
    Tree4<16, true> tree;
    for (int b = 0; b < B; ++b) tree.push(make_uint4(row_loss[b], 0, 0, 0));
    const uint4 acc = tree.finish(levels);
    *loss = (uint16_t)hmul2_rn(acc.x, dup2(ratio));
  }
}

cudaError_t launch_softmax_xent(const uint16_t* logits, const uint16_t* bias,
                                const int32_t* labels, int B, int K, uint16_t* loss,
                                uint16_t* dlogits, uint16_t* dbias, uint16_t* ws,
                                cudaStream_t s) {
  const uint16_t invB = f16_bits_host((float)(1.0 / B));
  int L = 0;
  while ((1 << L) < B) ++L;
  const uint16_t ratio = f16_bits_host((float)((double)(1 << L) / B));
  k_softmax_rows<<<B, kSmThreads, 0, s>>>(logits, bias, labels, K, invB, dlogits, ws);
  k_softmax_cols<<<(K + 255) / 256, 256, 0, s>>>(dlogits, ws, B, K, L, ratio, dbias, loss);
  return cudaGetLastError();
}

}  // namespace pf16
