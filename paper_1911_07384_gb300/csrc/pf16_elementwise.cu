// Memory-bound kernels of the pure-FP16 ResNet-50 training step: the FP16
// SGD-momentum update, BatchNorm forward/backward with the x0.25 output
// scaling, the split-K FP16 tree reduction of the weight gradient, the stem's
// patch gather, pooling and softmax cross-entropy.  All arithmetic is binary16
// (paper Sec. 5.2), one IEEE rounding per op (add.rn / mul.rn / sub.rn on
// f16x2, never contracted), subnormals kept.  Global traffic is 128-bit.
#include <cuda_fp16.h>

#include <cstring>

#include "../../include/pf16.h"
#include "pf16_internal.h"
#include "pf16_ptx.cuh"

namespace pf16 {

namespace {

constexpr uint32_t kHalfHalf2 = 0x38003800u;  // {0.5, 0.5}

__host__ __device__ __forceinline__ uint32_t dup2(uint16_t h) { return (uint32_t)h | ((uint32_t)h << 16); }

__device__ __forceinline__ uint4 add4(uint4 a, uint4 b) {
  return make_uint4(hadd2_rn(a.x, b.x), hadd2_rn(a.y, b.y), hadd2_rn(a.z, b.z), hadd2_rn(a.w, b.w));
}
// halving merge, the mean of two nodes: rn(a/2 + rn(b/2)) as one fused
// multiply-add.  It equals rn(rn(a/2) + rn(b/2)) whenever a/2 is exact (every
// a but a subnormal with its last bit set) and, halving before adding, never
// overflows.
__device__ __forceinline__ uint32_t hmerge2(uint32_t a, uint32_t b) {
  return hfma2_rn(a, kHalfHalf2, hmul2_rn(b, kHalfHalf2));
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

// x * 2^-e for e >= 0 by power-of-two steps: exact while the result is
// normal; a subnormal result is rounded (at most twice, once per step below
// 2^-14)
__device__ __forceinline__ uint4 ldexp_down4(uint4 v, int e) {
  while (e > 14) {
    v = mul4(v, dup2(0x0400));  // 2^-14
    e -= 14;
  }
  const uint16_t pe = (uint16_t)((15 - e) << 10);  // 2^-e, 0 <= e <= 14
  return mul4(v, dup2(pe));
}


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
  pdl_wait();
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
  launch_pdl(k_sgd, dim3((unsigned)blocks), dim3(256), 0, s, w, v, g, n, dup2(lr), dup2(mom), dup2(wd), wd != 0);
  return counted_launches(1);
}

// ============================================================================
// Data-parallel gradient exchange, combining step: out = rn(T * scale), T the
// perfect pairwise FP16 tree over `world` planes in plane order (padded with
// +0 leaves to a power of two).  Each thread owns one 8-element chunk: its
// leaves are loaded in aligned batches of up to 16 (all loads of a batch in
// flight), each batch summed as a perfect tree, and the batch sums merged by
// a register-resident binary counter -- together the perfect tree over the
// padded leaves.  Every load of a chunk precedes its store, so out may be
// plane 0.
// ============================================================================
__global__ void __launch_bounds__(256)
    k_dp_combine(const uint16_t* __restrict__ planes, int world, int world_pow2, long long nvec,
                 long long pstride_vec, uint32_t scale2, int do_scale, uint16_t* out) {
  pdl_wait();
  const uint4* P = reinterpret_cast<const uint4*>(planes);
  uint4* O = reinterpret_cast<uint4*>(out);
  const int nb = world_pow2 < 16 ? world_pow2 : 16;
  const long long step = (long long)gridDim.x * blockDim.x;
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < nvec; i += step) {
    uint4 st[7];  // st[l]: a finished subtree of 2^l batch sums (1024 / 16 = 2^6 batches at most)
    unsigned cnt = 0;
    for (int j0 = 0; j0 < world_pow2; j0 += 16) {
      uint4 v[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const int r = j0 + j;
        v[j] = (j < nb && r < world) ? P[(long long)r * pstride_vec + i] : zero4();
      }
#pragma unroll
      for (int w = 1; w < 16; w *= 2)
#pragma unroll
        for (int j = 0; j < 16; j += 2 * w)
          if (j + w < nb) v[j] = add4(v[j], v[j + w]);
      uint4 b = v[0];
      bool carry = true;
#pragma unroll
      for (int l = 0; l < 7; ++l) {
        const bool bit = (cnt >> l) & 1u;
        if (carry && bit) b = add4(st[l], b);
        if (carry && !bit) {
          st[l] = b;
          carry = false;
        }
      }
      ++cnt;
    }
    uint4 acc = zero4();
#pragma unroll
    for (int l = 0; l < 7; ++l)
      if (cnt == (1u << l)) acc = st[l];
    O[i] = do_scale ? mul4(acc, scale2) : acc;
  }
}

cudaError_t launch_dp_combine(const uint16_t* planes, int world, size_t n, size_t plane_stride, uint16_t scale,
                              uint16_t* out, cudaStream_t s) {
  int w2 = 1;
  while (w2 < world) w2 *= 2;
  const long long nvec = (long long)(n / 8);
  long long blocks = (nvec + 255) / 256;
  if (blocks > 152ll * 8) blocks = 152ll * 8;
  if (blocks < 1) blocks = 1;
  const uint32_t scale2 = (uint32_t)scale | ((uint32_t)scale << 16);
  launch_pdl(k_dp_combine, dim3((unsigned)blocks), dim3(256), 0, s, planes, world, w2, nvec,
             (long long)(plane_stride / 8), scale2, scale != 0x3C00 ? 1 : 0, out);
  return counted_launches(1);
}

// ============================================================================
// Split-K weight-gradient reduction: out = balanced pairwise FP16 tree over
// the `splits` partial matrices.
// ============================================================================
// A CTA of 256 threads = cl output chunks (8 columns each) x grp split groups;
// each thread sums a contiguous power-of-two run of splits (zero past the
// last split) with batched independent loads, then the groups are summed
// pairwise in shared memory: a balanced tree over the padded splits.
__global__ void __launch_bounds__(256)
    k_splitk_reduce(const uint16_t* __restrict__ parts, int splits, int splits_pow2, int grp,
                    long long rows, int cols, uint16_t* __restrict__ out, long long ldo,
                    int cols_out) {
  pdl_wait();
  __shared__ uint4 sh[256];
  const int cl = 256 / grp;
  const int t = threadIdx.x;
  const int lane = t % cl, g = t / cl;
  const int cpr = cols / 8;
  const long long total = rows * cpr;
  const long long chunk = (long long)blockIdx.x * cl + lane;
  const long long plane = rows * (long long)cols / 8;  // uint4 per partial plane
  const int seg = splits_pow2 / grp;
  uint4 acc = zero4();
  if (chunk < total) {
    const long long r = chunk / cpr;
    const int cg = (int)(chunk - r * cpr);
    const uint4* src = reinterpret_cast<const uint4*>(parts + r * cols + cg * 8);
    // seg is a power of two, so the run splits into aligned batches of
    // nb = min(seg, 16) leaves: each batch is summed as a perfect pairwise
    // tree with all its loads in flight at once, and the batch sums feed a
    // register-resident binary counter, which builds the perfect tree above
    // them.  Together: the perfect pairwise tree over the run's seg leaves.
    const int nb = seg < 16 ? seg : 16;
    uint4 st[8];  // st[l]: a finished subtree of 2^l batch sums
    unsigned cnt = 0;
    for (int i0 = 0; i0 < seg; i0 += 16) {
      uint4 v[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const int sp = g * seg + i0 + i;
        v[i] = (i < nb && sp < splits) ? __ldg(src + sp * plane) : zero4();
      }
#pragma unroll
      for (int w = 1; w < 16; w *= 2)
#pragma unroll
        for (int i = 0; i < 16; i += 2 * w)
          if (i + w < nb) v[i] = add4(v[i], v[i + w]);
      uint4 b = v[0];
      bool carry = true;
#pragma unroll
      for (int l = 0; l < 8; ++l) {
        const bool bit = (cnt >> l) & 1u;
        if (carry && bit) b = add4(st[l], b);
        if (carry && !bit) { st[l] = b; carry = false; }
      }
      ++cnt;
    }
    // cnt = seg / nb is a power of two: its one set bit names the full tree
#pragma unroll
    for (int l = 0; l < 8; ++l)
      if (cnt == (1u << l)) acc = st[l];
  }
  sh[t] = acc;
  __syncthreads();
  for (int half = grp / 2; half >= 1; half /= 2) {
    if (g < half) sh[t] = add4(sh[t], sh[t + half * cl]);
    __syncthreads();
  }
  if (g == 0 && chunk < total) {
    const long long r = chunk / cpr;
    const int cg = (int)(chunk - r * cpr);
    const uint4 v = sh[t];
    const uint16_t* h = reinterpret_cast<const uint16_t*>(&v);
    uint16_t* o = out + r * ldo + cg * 8;
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (cg * 8 + j < cols_out) o[j] = h[j];
  }
}

cudaError_t launch_splitk_reduce(const uint16_t* parts, int splits, long long rows, int cols,
                                 uint16_t* out, long long ldo, int cols_out, cudaStream_t s) {
  int sp2 = 1;
  while (sp2 < splits) sp2 *= 2;
  // Split groups per output chunk: only as many as it takes to give the GPU
  // about 512 threads per SM (one wave), each with up to 16 loads in flight,
  // so that a thread sums a long run of splits instead of each CTA paying a
  // shared-memory tree for a few loads.  Every choice sums the same balanced
  // tree over the padded splits.
  const long long total_chunks = rows * (cols / 8);
  int grp = 1;
  while (grp < sp2 && grp < 256 && total_chunks * grp < 152ll * 512) grp *= 2;
  const int cl = 256 / grp;
  const long long total = rows * (cols / 8);
  const long long blocks = (total + cl - 1) / cl;
  launch_pdl(k_splitk_reduce, dim3((unsigned)blocks), dim3(256), 0, s, parts, splits, sp2, grp, rows, cols, out, ldo, cols_out);
  return counted_launches(1);
}

// ============================================================================
// Stem patch gather (c = 3 cannot be fetched by TMA efficiently: a pixel is 6
// bytes).  col[m][j], m = (n, p, q), j = (r*S + s)*C + c < R*S*C, zero-padded
// to kcol.  One CTA per output row (n, p): the R input rows it needs are
// staged in shared memory with `pad` zero pixels on each side.  The CTA's
// output is Q * kcol contiguous halves; thread t owns the 16-byte piece
// g = t % G (G = kcol / 8) of pixels q = t / G, t / G + T / G, ..., so a warp
// stores consecutive 16-byte pieces and the thread's 8 source offsets stay in
// registers.
// ============================================================================
__global__ void k_stem_im2col(const uint16_t* __restrict__ x, uint16_t* __restrict__ col, int N,
                              int H, int W, int P, int Q, int R, int S, int C, int stride, int pad,
                              int kcol) {
  pdl_wait();
  extern __shared__ uint16_t rows[];  // [R][W + 2 pad][C]
  const int WP = W + 2 * pad;
  const int rowlen = WP * C;
  const int n = blockIdx.x / P, p = blockIdx.x - n * P;
  const int kin = R * S * C;
  const int G = kcol / 8;
  for (int r = 0; r < R; ++r) {
    const int h = p * stride + r - pad;
    uint16_t* dst = rows + r * rowlen;
    for (int e = threadIdx.x; e < pad * C; e += blockDim.x) {
      dst[e] = 0;
      dst[rowlen - 1 - e] = 0;
    }
    if (h < 0 || h >= H) {
      for (int e = threadIdx.x; e < W * C; e += blockDim.x) dst[pad * C + e] = 0;
      continue;
    }
    const uint16_t* src = x + ((long long)n * H + h) * W * C;
    if ((W * C) % 8 == 0) {  // every input row then starts 16-byte aligned
      for (int v = threadIdx.x; v < W * C / 8; v += blockDim.x) {
        const uint4 u = __ldg(reinterpret_cast<const uint4*>(src) + v);
        const uint16_t* hv = reinterpret_cast<const uint16_t*>(&u);
#pragma unroll
        for (int e = 0; e < 8; ++e) dst[pad * C + v * 8 + e] = hv[e];
      }
    } else {
      for (int e = threadIdx.x; e < W * C; e += blockDim.x) dst[pad * C + e] = src[e];
    }
  }
  __syncthreads();
  const int g = threadIdx.x % G;
  const int q0 = threadIdx.x / G, qs = blockDim.x / G;
  if (q0 >= qs) return;  // threads past the last whole group of G
  int off[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    const int j = g * 8 + e;
    const int c = j % C, rs = j / C;
    off[e] = j < kin ? (rs / S) * rowlen + (rs % S) * C + c : -1;
  }
  uint4* out = reinterpret_cast<uint4*>(col + (long long)blockIdx.x * Q * kcol);
  for (int q = q0; q < Q; q += qs) {
    const uint16_t* base = rows + q * stride * C;
    uint32_t v[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const uint32_t lo = off[2 * e] >= 0 ? base[off[2 * e]] : 0u;
      const uint32_t hi = off[2 * e + 1] >= 0 ? base[off[2 * e + 1]] : 0u;
      v[e] = lo | (hi << 16);
    }
    out[(long long)q * G + g] = make_uint4(v[0], v[1], v[2], v[3]);
  }
}

cudaError_t launch_stem_im2col(const uint16_t* x, uint16_t* col, int N, int H, int W, int P, int Q,
                               int R, int S, int C, int stride, int pad, int kcol,
                               cudaStream_t s) {
  const size_t shm = (size_t)R * (W + 2 * pad) * C * sizeof(uint16_t);
  if (shm > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(k_stem_im2col, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)shm);
    if (e != cudaSuccess) return e;
  }
  // a whole number of G-thread groups, about 160 threads, in whole warps
  const int G = kcol / 8;
  int threads = G * ((160 + G - 1) / G);
  if (threads > 1024) threads = G;
  threads = (threads + 31) / 32 * 32;
  launch_pdl(k_stem_im2col, dim3((unsigned)((long long)N * P)), dim3(threads), shm, s, x, col, N, H, W, P, Q, R, S, C, stride,
                                                                   pad, kcol);
  return counted_launches(1);
}

// ============================================================================
// Stem space-to-depth (7x7 / stride 2 / pad 3 over 3 channels becomes a 4x4 /
// stride 1 convolution over 16 channels):
//   xs[n][I][J][(a*2 + b)*4 + c] = x[n][2I + a - 3][2J + b - 3][c]   (c < 3),
//   0 for c = 3 and outside x;  I < Hs, J < Ws;
//   wsd[k][(u*4 + v)*16 + (a*2 + b)*4 + c] = w[k][2u + a][2v + b][c],
//   0 for c = 3 or where 2u + a or 2v + b reaches 7.
// Blocks below N*Hs each write one row (n, I) of xs from the two input rows
// 2I - 3, 2I - 2 staged in shared memory, one 32-byte pixel per thread (a
// warp stores 1 KB contiguous); the blocks after them pack the filter.
// ============================================================================
__global__ void k_stem_s2d(const uint16_t* __restrict__ x, const uint16_t* __restrict__ w,
                           uint16_t* __restrict__ xs, uint16_t* __restrict__ wsd, int N, int H, int W,
                           int Hs, int Ws, int K) {
  pdl_wait();
  const long long rows_total = (long long)N * Hs;
  if ((long long)blockIdx.x >= rows_total) {
    const int e = (int)(blockIdx.x - rows_total) * blockDim.x + threadIdx.x;
    if (e >= K * 256) return;
    const int k = e >> 8, j = e & 255;
    const int t = j >> 4, ch = j & 15;
    const int r = 2 * (t >> 2) + (ch >> 3), sc = 2 * (t & 3) + ((ch >> 2) & 1), c = ch & 3;
    wsd[e] = (c < 3 && r < 7 && sc < 7) ? w[((k * 7 + r) * 7 + sc) * 3 + c] : (uint16_t)0;
    return;
  }
  extern __shared__ uint16_t srow[];  // [2][W * 3]
  const int n = (int)(blockIdx.x / Hs), I = (int)(blockIdx.x - (long long)n * Hs);
  const int len = W * 3;
  for (int a = 0; a < 2; ++a) {
    const int h = 2 * I + a - 3;
    uint16_t* dst = srow + a * len;
    if (h < 0 || h >= H) {
      for (int e = threadIdx.x; e < len; e += blockDim.x) dst[e] = 0;
      continue;
    }
    const uint16_t* src = x + ((long long)n * H + h) * len;
    if (len % 8 == 0) {  // every input row then starts 16-byte aligned
      for (int v = threadIdx.x; v < len / 8; v += blockDim.x) {
        const uint4 u = __ldg(reinterpret_cast<const uint4*>(src) + v);
        *reinterpret_cast<uint4*>(dst + v * 8) = u;
      }
    } else {
      for (int e = threadIdx.x; e < len; e += blockDim.x) dst[e] = src[e];
    }
  }
  __syncthreads();
  uint4* out = reinterpret_cast<uint4*>(xs + ((long long)n * Hs + I) * Ws * 16);
  for (int J = threadIdx.x; J < Ws; J += blockDim.x) {
    uint32_t v[8];
#pragma unroll
    for (int a = 0; a < 2; ++a)
#pragma unroll
      for (int b = 0; b < 2; ++b) {
        const int col = 2 * J + b - 3;
        uint32_t c0 = 0, c1 = 0, c2 = 0;
        if (col >= 0 && col < W) {
          const uint16_t* q = srow + a * len + col * 3;
          c0 = q[0];
          c1 = q[1];
          c2 = q[2];
        }
        v[(a * 2 + b) * 2] = c0 | (c1 << 16);
        v[(a * 2 + b) * 2 + 1] = c2;
      }
    out[(long long)J * 2] = make_uint4(v[0], v[1], v[2], v[3]);
    out[(long long)J * 2 + 1] = make_uint4(v[4], v[5], v[6], v[7]);
  }
}

cudaError_t launch_stem_s2d(const uint16_t* x, const uint16_t* w, uint16_t* xs, uint16_t* wsd, int N, int H,
                            int W, int Hs, int Ws, int K, cudaStream_t s) {
  const size_t shm = (size_t)2 * W * 3 * sizeof(uint16_t);
  if (shm > 48 * 1024) return cudaErrorInvalidValue;
  const int threads = 128;
  const long long blocks = (long long)N * Hs + (K * 256 + threads - 1) / threads;
  if (blocks > 0x7fffffffll) return cudaErrorInvalidValue;
  launch_pdl(k_stem_s2d, dim3((unsigned)blocks), dim3(threads), shm, s, x, w, xs, wsd, N, H, W, Hs, Ws, K);
  return counted_launches(1);
}

// dws[row][col], row = 64 (tap row even) or 0 (odd) + k, col = (tap row / 2) * 64
// + (tap column) * 16 + (a*2 + b)*4 + c, for r = 2 * tap row + a, s = 2 * tap
// column + b (the stem weight gradient's layout) -> dw[k][r][s][c], 7 x 7 x 3
__global__ void k_stem_wgrad_scatter(const uint16_t* __restrict__ dws, uint16_t* __restrict__ dw, int K) {
  pdl_wait();
  const int e = blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= K * 147) return;
  const int k = e / 147, rsc = e - k * 147;
  const int r = rsc / 21, sc = rsc - r * 21, sx = sc / 3, c = sc - sx * 3;
  const int tr = r >> 1, tc = sx >> 1;
  const int row = ((tr & 1) ? 0 : 64) + k;
  const int col = (tr >> 1) * 64 + tc * 16 + ((r & 1) * 2 + (sx & 1)) * 4 + c;
  dw[e] = dws[row * 128 + col];
}

cudaError_t launch_stem_wgrad_scatter(const uint16_t* dws, uint16_t* dw, int K, cudaStream_t s) {
  if (K != 64) return cudaErrorInvalidValue;
  launch_pdl(k_stem_wgrad_scatter, dim3((K * 147 + 255) / 256), dim3(256), 0, s, dws, dw, K);
  return counted_launches(1);
}

__global__ void k_pad_rows(const uint16_t* __restrict__ w, uint16_t* __restrict__ wp, int K, int kin,
                           int kcol) {
  pdl_wait();
  const int total = K * kcol;
  for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < total; t += gridDim.x * blockDim.x) {
    const int k = t / kcol, j = t - k * kcol;
    wp[t] = j < kin ? w[k * kin + j] : (uint16_t)0;
  }
}

cudaError_t launch_pad_rows(const uint16_t* w, uint16_t* wp, int K, int kin, int kcol,
                            cudaStream_t s) {
  const int blocks = (K * kcol + 255) / 256;
  launch_pdl(k_pad_rows, dim3(blocks), dim3(256), 0, s, w, wp, K, kin, kcol);
  return counted_launches(1);
}

cudaError_t launch_fill_zero(uint16_t* p, size_t n, cudaStream_t s) {
  return cudaMemsetAsync(p, 0, n * sizeof(uint16_t), s);
}

// ============================================================================
// BatchNorm (Eq. 1, Eq. 2, then x post_scale, + residual, ReLU), FP16 only.
//
// Statistics are balanced pairwise trees over the R rows of each channel.
// Rows come in chunks of RB = rpb * 8 consecutive rows, which are contiguous
// in memory; a statistics CTA owns chunks b, b + grid, b + 2 grid, ... (so
// consecutive CTAs stream adjacent rows).  Its producer warp streams them
// through a ring of shared-memory stages with one bulk copy per tensor per
// chunk, so the bytes in flight are set by the ring, not by registers; its
// consumer threads each reduce 8 rows (strided by rpb) of one group of 8
// channels per chunk from shared memory:
//   forward:  per chunk the mean of the thread's valid rows and the mean
//             squared deviation from it (register trees over the 8 rows: x is
//             read once), merged over the thread's chunks and then over the
//             CTA's row groups by the count-aware pairwise parallel-variance
//             rule;
//   backward: the pairwise sums of dy' and dy' * xhat over the 8 rows, a
//             pairwise tree over the thread's chunks, then over the CTA's row
//             groups (zero padded to powers of two throughout).
// A second small kernel (one CTA per channel group) combines the per-CTA
// results over a balanced tree: forward by the parallel-variance rule (exact
// counts), backward by pairwise sum trees: dgamma and dbeta are the sums x
// post_scale, the means rn(rn(sum * rn(2^L/R)) * 2^-L).  (Sums, not halving
// means: gradients are small, and halving a subnormal partial mean drops its
// low bits -- in the last stage of the batch-256 step that lost the whole of
// dbeta.)  Then one elementwise pass applies.  With ReLU the forward can also
// store the ReLU decisions as a bit mask, which the backward then reads in
// place of the saved output (1/16 of its bytes).
// ============================================================================
namespace {

constexpr int kBnThreads = 256;                 // consumer threads per CTA, at most
constexpr int kStatRowsT = 8;                   // rows per consumer thread per chunk
constexpr int kStatStages = 3;                  // shared-memory ring depth
constexpr int kStatLevels = 9;                  // per-thread chunk trees: up to 256 chunks
constexpr int kStatMaxChunks = 1 << (kStatLevels - 1);
constexpr int kStatTensorBytes = kStatRowsT * kBnThreads * 16;  // one tensor's slot: RB rows <= 32 KB
constexpr int kFwdCtasPerSm = 2;                // forward ring: 3 x 32 KB (x)
constexpr int kBwdCtasPerSm = 1;                // backward ring: 3 x 64 KB (x, dy)
constexpr int kGb300Sms = 152;

struct BnGeom {
  int tc;       // threads per row: channel groups of 8
  int rpb;      // row groups per CTA (power of two, at most 32)
  int threads;  // tc * rpb rounded up to whole warps
};

__host__ __device__ inline BnGeom bn_geom(int C) {
  BnGeom g;
  g.tc = C / 8;
  int rpb = 1;
  while (rpb < 32 && rpb * 2 * g.tc <= kBnThreads) rpb *= 2;
  g.rpb = rpb;
  g.threads = (g.tc * rpb + 31) / 32 * 32;
  return g;
}

__host__ __device__ constexpr int stat_smem_bytes(int ntensor) {
  return kStatStages * ntensor * kStatTensorBytes + 16 * kStatStages;
}

struct BnStatArgs {
  const uint16_t* x;
  const uint16_t* dy;
  const uint16_t* y_saved;    // backward, ReLU from the saved output
  const uint8_t* mask_in;     // backward, ReLU from the bit mask
  const uint16_t* mean_in;    // backward: saved mean
  const uint16_t* invstd_in;  // backward: saved invstd
  int R, C, blocks, blocks_pow2;
  int mean_levels;      // backward: ceil(log2 R); mean = (sum * ratio) * 2^-mean_levels
  int chunk_levels;     // the CTA's per-thread chunk trees are padded to 2^chunk_levels
  uint16_t ratio;       // backward: rn(2^mean_levels / R), in [1, 2)
  uint16_t eps, post_scale;
  int* status;          // device status word
  unsigned long long wait_limit_ns;
  uint16_t* ws1;        // [blocks][C]
  uint16_t* ws2;        // [blocks][C]
  // outputs
  uint16_t* mean_out;
  uint16_t* invstd_out;
  uint16_t* dgamma;
  uint16_t* dbeta;
  uint16_t* mm;         // backward: mean(dy'), mean(dy' xhat) for the apply pass, [2][C]
  uint16_t* ws4;        // backward, swap variant: per-CTA trees of dy' * residual [blocks][C], else null
};

__device__ __forceinline__ uint4 tree8(uint4* v) {
#pragma unroll
  for (int w = 4; w >= 1; w /= 2)
#pragma unroll
    for (int i = 0; i < w; ++i) v[i] = hmerge4(v[2 * i], v[2 * i + 1]);
  return v[0];
}
// the pairwise sum of 8 rows (backward statistics)
__device__ __forceinline__ uint4 sum8(uint4* v) {
#pragma unroll
  for (int w = 4; w >= 1; w /= 2)
#pragma unroll
    for (int i = 0; i < w; ++i) v[i] = add4(v[2 * i], v[2 * i + 1]);
  return v[0];
}

__device__ __forceinline__ uint4 and4(uint4 a, uint4 m) {
  return make_uint4(a.x & m.x, a.y & m.y, a.z & m.z, a.w & m.w);
}
// per-lane all-ones where the saved output is > 0 (the ReLU passed)
__device__ __forceinline__ uint4 relu_mask4(uint4 y) {
  return make_uint4(relu_mask2(y.x), relu_mask2(y.y), relu_mask2(y.z), relu_mask2(y.w));
}
// the two lane bits of a per-lane all-ones mask
__device__ __forceinline__ uint32_t mask_bits2(uint32_t m) { return (m & 1u) | ((m >> 15) & 2u); }
// ReLU of z, and the decisions as bits (bit j: lane j of z is > 0)
__device__ __forceinline__ uint4 relu_bits(uint4 z, uint32_t& bits) {
  const uint4 m = relu_mask4(z);
  bits = mask_bits2(m.x) | mask_bits2(m.y) << 2 | mask_bits2(m.z) << 4 | mask_bits2(m.w) << 6;
  return and4(z, m);
}
__device__ __forceinline__ uint32_t bits_mask2(uint32_t b) {
  return ((b & 1u) ? 0x0000FFFFu : 0u) | ((b & 2u) ? 0xFFFF0000u : 0u);
}
__device__ __forceinline__ uint4 bits_mask4(uint32_t b) {
  return make_uint4(bits_mask2(b), bits_mask2(b >> 2), bits_mask2(b >> 4), bits_mask2(b >> 6));
}

// Combination of (mean, variance) pairs by the pairwise parallel variance
// rule: merging groups a and b with counts na, nb gives
//   mean = wa*mean_a + wb*mean_b,  var = wa*var_a + wb*var_b + wa*wb*(mean_b - mean_a)^2,
// wa = na/(na+nb).  For equal counts this is exactly the halving merge of the
// means and of the variances plus ((mean_b - mean_a)/2)^2.  Weights are
// constants of the counts.
struct MV {
  uint4 mu, v;
  long long n;
};

__device__ __forceinline__ MV mv_merge(const MV& a, const MV& b) {
  if (b.n == 0) return a;
  if (a.n == 0) return b;
  MV r;
  r.n = a.n + b.n;
  const uint4 d = sub4(b.mu, a.mu);
  if (a.n == b.n) {
    r.mu = hmerge4(a.mu, b.mu);
    const uint4 dh = mul4(d, kHalfHalf2);
    r.v = add4(hmerge4(a.v, b.v), mul4v(dh, dh));
  } else {
    // weights in binary32 (exact count ratios to 2^-24), then rounded to binary16
    const __half wa = __float2half_rn(__fdiv_rn((float)a.n, (float)r.n));
    const __half wb = __float2half_rn(__fdiv_rn((float)b.n, (float)r.n));
    const uint32_t wa2 = dup2(__half_as_ushort(wa)), wb2 = dup2(__half_as_ushort(wb));
    const uint32_t wab2 = hmul2_rn(wa2, wb2);
    r.mu = add4(mul4(a.mu, wa2), mul4(b.mu, wb2));
    r.v = add4(add4(mul4(a.v, wa2), mul4(b.v, wb2)), mul4(mul4v(d, d), wab2));
  }
  return r;
}

// Barrier over the consumer warps only (the producer warp may have left).
__device__ __forceinline__ void consumers_sync(int n) {
  asm volatile("bar.sync 1, %0;" ::"r"(n) : "memory");
}

// Producer (one lane): stream the CTA's chunks through the ring.  Stage s of
// chunk ci is refilled only after every consumer warp has released it.  On a
// wait that runs out it records the timeout and lets the copies it already
// issued land before returning.
__device__ __noinline__ void stat_produce(const BnStatArgs& a, long long RB, uint32_t ring, uint32_t bars,
                                          int ntensor, const uint16_t* t0, const uint16_t* t1) {
  const long long rowb = 2ll * a.C;
  const uint32_t stage_bytes = (uint32_t)(ntensor * kStatTensorBytes);
  int ci = 0;
  bool ok = true;
  for (;; ++ci) {
    const long long row0 = ((long long)ci * gridDim.x + blockIdx.x) * RB;
    if (row0 >= a.R) break;
    const int s = ci % kStatStages;
    const uint32_t full = bars + 8 * s, empty = bars + 8 * (kStatStages + s);
    if (ci >= kStatStages && !mbar_wait(empty, (uint32_t)((ci / kStatStages - 1) & 1), a.wait_limit_ns)) {
      ok = false;
      break;
    }
    const long long rows = a.R - row0 < RB ? a.R - row0 : RB;
    const uint32_t bytes = (uint32_t)(rows * rowb);
    const uint32_t dst = ring + (uint32_t)s * stage_bytes;
    mbar_arrive_expect_tx(full, bytes * (uint32_t)ntensor);
    bulk_load_1d(dst, t0 + row0 * a.C, bytes, full);
    if (ntensor == 2) bulk_load_1d(dst + kStatTensorBytes, t1 + row0 * a.C, bytes, full);
  }
  if (!ok) {
    atomicExch(a.status, PF16_ERR_TIMEOUT);
    for (int c = ci - kStatStages < 0 ? 0 : ci - kStatStages; c < ci; ++c)
      mbar_wait(bars + 8 * (c % kStatStages), (uint32_t)((c / kStatStages) & 1), a.wait_limit_ns);
  }
}

// Ring set-up shared by both statistics kernels; returns the barrier base.
__device__ __forceinline__ uint32_t stat_ring_init(uint32_t ring, int ntensor, int ncons) {
  const uint32_t bars = ring + (uint32_t)(kStatStages * ntensor * kStatTensorBytes);
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStatStages; ++s) {
      mbar_init(bars + 8 * s, 1);                            // full: the producer's expect_tx
      mbar_init(bars + 8 * (kStatStages + s), ncons / 32);   // empty: one arrival per consumer warp
    }
    fence_mbar_init();
  }
  __syncthreads();
  return bars;
}

// Forward statistics.  Consumers: cg = t % tc (a warp reads consecutive 16-byte
// columns of a row from shared memory), rg = t / tc.
__global__ void __launch_bounds__(kBnThreads + 32, kFwdCtasPerSm) k_bn_fwd_stats(const BnStatArgs a) {
  pdl_wait();
  extern __shared__ __align__(128) uint8_t stat_smem[];
  __shared__ uint4 smu[kBnThreads], sv[kBnThreads];
  __shared__ long long sn[kBnThreads];
  const BnGeom g = bn_geom(a.C);
  const int t = threadIdx.x, ncons = g.threads;
  const uint32_t ring = smem_u32(stat_smem);
  const uint32_t bars = stat_ring_init(ring, 1, ncons);
  const long long RB = (long long)g.rpb * kStatRowsT;
  if (t >= ncons) {
    if (t == ncons) stat_produce(a, RB, ring, bars, 1, a.x, nullptr);
    return;
  }
  const int cg = t % g.tc, rg = t / g.tc;
  const bool active = t < g.tc * g.rpb;
  MV st[kStatLevels];
  unsigned cnt = 0;
  bool ok = true;
  for (int ci = 0;; ++ci) {
    const long long row0 = ((long long)ci * gridDim.x + blockIdx.x) * RB;
    if (row0 >= a.R) break;
    const int s = ci % kStatStages;
    if (!mbar_wait(bars + 8 * s, (uint32_t)((ci / kStatStages) & 1), a.wait_limit_ns)) {
      ok = false;
      break;
    }
    const uint32_t base = ring + (uint32_t)s * kStatTensorBytes;
    uint4 v[kStatRowsT], d[kStatRowsT];
    int nv = 0;
#pragma unroll
    for (int i = 0; i < kStatRowsT; ++i) {
      const int r = rg + i * g.rpb;
      const bool okr = active && row0 + r < a.R;  // valid rows are a prefix of the thread's 8
      nv += okr;
      v[i] = zero4();
      if (okr) ld_shared_v4(base + (uint32_t)(r * g.tc + cg) * 16u, v[i]);
      d[i] = v[i];
    }
    __syncwarp();
    if ((t & 31) == 0) mbar_arrive(bars + 8 * (kStatStages + s));
    if (nv == 0) continue;
    // mean of the valid rows: padded halving tree, rescaled when rows are missing
    uint4 mu = tree8(d);
    uint32_t sc = 0;
    if (nv < kStatRowsT) {
      sc = dup2(__half_as_ushort(__float2half_rn((float)kStatRowsT / (float)nv)));
      mu = mul4(mu, sc);
    }
#pragma unroll
    for (int i = 0; i < kStatRowsT; ++i) {
      const uint4 e = sub4(v[i], mu);
      d[i] = (i < nv) ? mul4v(e, e) : zero4();
    }
    uint4 var = tree8(d);
    if (nv < kStatRowsT) var = mul4(var, sc);
    MV node{mu, var, nv};
#pragma unroll 1
    for (int l = 0; l < kStatLevels; ++l) {
      if (cnt & (1u << l)) {
        node = mv_merge(st[l], node);
      } else {
        st[l] = node;
        break;
      }
    }
    ++cnt;
  }
  if (!ok) atomicExch(a.status, PF16_ERR_TIMEOUT);
  MV acc{zero4(), zero4(), 0};
#pragma unroll 1
  for (int l = 0; l < kStatLevels; ++l)
    if (cnt & (1u << l)) acc = mv_merge(st[l], acc);
  smu[t] = acc.mu;
  sv[t] = acc.v;
  sn[t] = acc.n;
  consumers_sync(ncons);
  for (int half = g.rpb / 2; half >= 1; half /= 2) {
    if (active && rg < half) {
      const int o = (rg + half) * g.tc + cg;
      const MV r = mv_merge(MV{smu[t], sv[t], sn[t]}, MV{smu[o], sv[o], sn[o]});
      smu[t] = r.mu;
      sv[t] = r.v;
      sn[t] = r.n;
    }
    consumers_sync(ncons);
  }
  if (active && rg == 0) {
    reinterpret_cast<uint4*>(a.ws1)[(long long)blockIdx.x * g.tc + cg] = smu[t];
    reinterpret_cast<uint4*>(a.ws2)[(long long)blockIdx.x * g.tc + cg] = sv[t];
  }
}

// ReLU source of the backward kernels
enum BnRelu : int { BN_NO_RELU = 0, BN_RELU_SAVED = 1, BN_RELU_BITS = 2 };

// Backward statistics, same consumer layout.  The ReLU decisions of the next
// chunk (bit-mask bytes, or saved-output vectors) are loaded from global
// memory while the current chunk is reduced.
// XRAW (the swap variant's second pass, x = the residual input): the second
// tree sums dy' * x itself instead of dy' * xhat.
template <int RELU, bool XRAW = false>
__global__ void __launch_bounds__(kBnThreads + 32, kBwdCtasPerSm) k_bn_bwd_stats(const BnStatArgs a) {
  pdl_wait();
  extern __shared__ __align__(128) uint8_t stat_smem[];
  __shared__ uint4 s1[kBnThreads], s2[kBnThreads];
  const BnGeom g = bn_geom(a.C);
  const int t = threadIdx.x, ncons = g.threads;
  const uint32_t ring = smem_u32(stat_smem);
  const uint32_t bars = stat_ring_init(ring, 2, ncons);
  const long long RB = (long long)g.rpb * kStatRowsT;
  if (t >= ncons) {
    if (t == ncons) stat_produce(a, RB, ring, bars, 2, a.x, a.dy);
    return;
  }
  const int cg = t % g.tc, rg = t / g.tc;
  const bool active = t < g.tc * g.rpb;
  uint4 mu = zero4(), is = zero4();
  if (active && !XRAW) {
    mu = __ldg(reinterpret_cast<const uint4*>(a.mean_in) + cg);
    is = __ldg(reinterpret_cast<const uint4*>(a.invstd_in) + cg);
  }
  // ReLU decisions of one chunk's rows of this thread
  uint32_t mb[kStatRowsT];
  uint4 ys[kStatRowsT];
  auto load_relu = [&](int ci) {
    const long long row0 = ((long long)ci * gridDim.x + blockIdx.x) * RB;
#pragma unroll
    for (int i = 0; i < kStatRowsT; ++i) {
      const long long r = row0 + rg + (long long)i * g.rpb;
      const bool okr = active && r < a.R;
      const long long off = r * g.tc + cg;
      if (RELU == BN_RELU_BITS) mb[i] = okr ? (uint32_t)__ldg(a.mask_in + off) : 0u;
      if (RELU == BN_RELU_SAVED) ys[i] = okr ? __ldg(reinterpret_cast<const uint4*>(a.y_saved) + off) : zero4();
    }
  };
  if (RELU != BN_NO_RELU) load_relu(0);
  uint4 st1[kStatLevels], st2[kStatLevels];
  unsigned cnt = 0;
  bool ok = true;
  for (int ci = 0;; ++ci) {
    const long long row0 = ((long long)ci * gridDim.x + blockIdx.x) * RB;
    if (row0 >= a.R) break;
    uint32_t mcur[kStatRowsT];
    uint4 ycur[kStatRowsT];
#pragma unroll
    for (int i = 0; i < kStatRowsT; ++i) {
      if (RELU == BN_RELU_BITS) mcur[i] = mb[i];
      if (RELU == BN_RELU_SAVED) ycur[i] = ys[i];
    }
    if (RELU != BN_NO_RELU) load_relu(ci + 1);  // rows past R are not read
    const int s = ci % kStatStages;
    if (!mbar_wait(bars + 8 * s, (uint32_t)((ci / kStatStages) & 1), a.wait_limit_ns)) {
      ok = false;
      break;
    }
    const uint32_t base = ring + (uint32_t)s * (2u * kStatTensorBytes);
    uint4 p1[kStatRowsT], p2[kStatRowsT];
#pragma unroll
    for (int i = 0; i < kStatRowsT; ++i) {
      const int r = rg + i * g.rpb;
      const bool okr = active && row0 + r < a.R;
      uint4 xv = zero4(), dv = zero4();
      if (okr) {
        const uint32_t o = (uint32_t)(r * g.tc + cg) * 16u;
        ld_shared_v4(base + o, xv);
        ld_shared_v4(base + kStatTensorBytes + o, dv);
      }
      if (RELU == BN_RELU_BITS) dv = and4(dv, bits_mask4(mcur[i]));
      if (RELU == BN_RELU_SAVED) dv = and4(dv, relu_mask4(ycur[i]));
      const uint4 xh = XRAW ? xv : mul4v(sub4(xv, mu), is);
      p1[i] = dv;
      p2[i] = okr ? mul4v(dv, xh) : zero4();
    }
    __syncwarp();
    if ((t & 31) == 0) mbar_arrive(bars + 8 * (kStatStages + s));
    uint4 n1 = sum8(p1), n2 = sum8(p2);
#pragma unroll 1
    for (int l = 0; l < kStatLevels; ++l) {
      if (cnt & (1u << l)) {
        n1 = add4(st1[l], n1);
        n2 = add4(st2[l], n2);
      } else {
        st1[l] = n1;
        st2[l] = n2;
        break;
      }
    }
    ++cnt;
  }
  if (!ok) atomicExch(a.status, PF16_ERR_TIMEOUT);
  // close the chunk trees as if zero chunks padded them to 2^chunk_levels
  uint4 acc1 = zero4(), acc2 = zero4();
  bool have = false;
#pragma unroll 1
  for (int l = 0; l < kStatLevels; ++l) {
    if (l < a.chunk_levels) {
      if (cnt & (1u << l)) {
        acc1 = add4(st1[l], have ? acc1 : zero4());
        acc2 = add4(st2[l], have ? acc2 : zero4());
        have = true;
      } else if (have) {
        acc1 = add4(acc1, zero4());
        acc2 = add4(acc2, zero4());
      }
    } else if (l == a.chunk_levels && (cnt & (1u << l))) {
      acc1 = st1[l];
      acc2 = st2[l];
    }
  }
  s1[t] = acc1;
  s2[t] = acc2;
  consumers_sync(ncons);
  for (int half = g.rpb / 2; half >= 1; half /= 2) {
    if (active && rg < half) {
      const int o = (rg + half) * g.tc + cg;
      s1[t] = add4(s1[t], s1[o]);
      s2[t] = add4(s2[t], s2[o]);
    }
    consumers_sync(ncons);
  }
  if (active && rg == 0) {
    reinterpret_cast<uint4*>(a.ws1)[(long long)blockIdx.x * g.tc + cg] = s1[t];
    reinterpret_cast<uint4*>(a.ws2)[(long long)blockIdx.x * g.tc + cg] = s2[t];
  }
}

constexpr int kFinalThreads = 256;
static_assert(kFinalThreads == kBnStatSlots, "the slot finals load one slot per thread");
__device__ __forceinline__ uint4 shfl_down4(uint4 v, int d) {
  return make_uint4(__shfl_down_sync(0xffffffffu, v.x, d), __shfl_down_sync(0xffffffffu, v.y, d),
                    __shfl_down_sync(0xffffffffu, v.z, d), __shfl_down_sync(0xffffffffu, v.w, d));
}

// One CTA per group of 8 channels: each thread merges a contiguous run of
// per-CTA results (loaded together), then the threads are merged in pairs in
// shared memory; both levels follow a balanced binary tree.  chunk_rows is RB;
// CTA b owns chunks b, b + blocks, ... and only the last chunk can be partial.
__global__ void __launch_bounds__(kFinalThreads) k_bn_fwd_final(const BnStatArgs a, long long chunk_rows) {
  pdl_wait();
  __shared__ uint4 smu[kFinalThreads], sv[kFinalThreads];
  __shared__ long long sn[kFinalThreads];
  const int tc = a.C / 8, cg = blockIdx.x, t = threadIdx.x;
  const int nthr = a.blocks_pow2 < kFinalThreads ? a.blocks_pow2 : kFinalThreads;
  const int seg = a.blocks_pow2 / nthr;
  const long long chunks = ((long long)a.R + chunk_rows - 1) / chunk_rows;
  const long long last_rows = (long long)a.R - (chunks - 1) * chunk_rows;
  const int last_owner = (int)((chunks - 1) % a.blocks);
  auto count = [&](int b) -> long long {
    if (b >= a.blocks) return 0;
    const long long nb = (chunks - b + a.blocks - 1) / a.blocks;
    return nb * chunk_rows - (b == last_owner ? chunk_rows - last_rows : 0);
  };
  if (t < nthr) {
    // binary-counter tree over this thread's seg slots (seg is a power of two)
    MV st[12];
    unsigned cnt = 0;
    for (int i0 = 0; i0 < seg; i0 += 4) {
      uint4 m[4], q[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int b = t * seg + i0 + i;
        const bool ok = (i0 + i < seg) && b < a.blocks;
        m[i] = ok ? __ldg(reinterpret_cast<const uint4*>(a.ws1) + (long long)b * tc + cg) : zero4();
        q[i] = ok ? __ldg(reinterpret_cast<const uint4*>(a.ws2) + (long long)b * tc + cg) : zero4();
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        if (i0 + i >= seg) break;
        MV node{m[i], q[i], count(t * seg + i0 + i)};
#pragma unroll
        for (int l = 0; l < 12; ++l) {
          if (cnt & (1u << l)) {
            node = mv_merge(st[l], node);
          } else {
            st[l] = node;
            break;
          }
        }
        ++cnt;
      }
    }
    const int lv = 31 - __clz(seg);  // seg == 2^lv, cnt == seg: the tree is st[lv]
    MV res = st[0];
#pragma unroll
    for (int l = 0; l < 12; ++l)
      if (l == lv) res = st[l];
    smu[t] = res.mu;
    sv[t] = res.v;
    sn[t] = res.n;
  }
  __syncthreads();
  for (int half = nthr / 2; half >= 1; half /= 2) {
    if (t < half) {
      const MV r = mv_merge(MV{smu[t], sv[t], sn[t]}, MV{smu[t + half], sv[t + half], sn[t + half]});
      smu[t] = r.mu;
      sv[t] = r.v;
      sn[t] = r.n;
    }
    __syncthreads();
  }
  if (t == 0) {
    const uint4 ve = add4(sv[0], make_uint4(dup2(a.eps), dup2(a.eps), dup2(a.eps), dup2(a.eps)));
    uint4 is;
    const __half2* hv = reinterpret_cast<const __half2*>(&ve);
    __half2* hi = reinterpret_cast<__half2*>(&is);
#pragma unroll
    for (int j = 0; j < 4; ++j) hi[j] = h2rsqrt(hv[j]);
    reinterpret_cast<uint4*>(a.mean_out)[cg] = smu[0];
    reinterpret_cast<uint4*>(a.invstd_out)[cg] = is;
  }
}

// Backward: pairwise sum trees over the per-CTA sums (zero padding is exact),
// then the sums scaled by post_scale (dbeta, dgamma) and the means
// rn(rn(sum * rn(2^L/R)) * 2^-L), L = ceil(log2 R).  Swap variant (a.ws4):
// dbeta = sum dy' (no post_scale) and dgamma = rn(rn(s * sum dy' xhat) +
// sum dy' r), the third tree over a.ws4.
__global__ void __launch_bounds__(kFinalThreads) k_bn_bwd_final(const BnStatArgs a) {
  pdl_wait();
  __shared__ uint4 s1[kFinalThreads], s2[kFinalThreads], s3[kFinalThreads];
  const int tc = a.C / 8, cg = blockIdx.x, t = threadIdx.x;
  const int nthr = a.blocks_pow2 < kFinalThreads ? a.blocks_pow2 : kFinalThreads;
  const int seg = a.blocks_pow2 / nthr;
  const bool swap = a.ws4 != nullptr;
  if (t < nthr) {
    Tree4<12, false> t1, t2, t3;
    for (int i0 = 0; i0 < seg; i0 += 4) {
      uint4 p[4], q[4], w[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int b = t * seg + i0 + i;
        const bool ok = (i0 + i < seg) && b < a.blocks;
        p[i] = ok ? __ldg(reinterpret_cast<const uint4*>(a.ws1) + (long long)b * tc + cg) : zero4();
        q[i] = ok ? __ldg(reinterpret_cast<const uint4*>(a.ws2) + (long long)b * tc + cg) : zero4();
        w[i] = (ok && swap) ? __ldg(reinterpret_cast<const uint4*>(a.ws4) + (long long)b * tc + cg) : zero4();
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        if (i0 + i >= seg) break;
        t1.push(p[i]);
        t2.push(q[i]);
        if (swap) t3.push(w[i]);
      }
    }
    const int lv = 31 - __clz(seg);
    s1[t] = t1.finish(lv);
    s2[t] = t2.finish(lv);
    s3[t] = swap ? t3.finish(lv) : zero4();
  }
  __syncthreads();
  for (int half = nthr / 2; half >= 1; half /= 2) {
    if (t < half) {
      s1[t] = add4(s1[t], s1[t + half]);
      s2[t] = add4(s2[t], s2[t + half]);
      if (swap) s3[t] = add4(s3[t], s3[t + half]);
    }
    __syncthreads();
  }
  if (t == 0) {
    const uint32_t ratio2 = dup2(a.ratio), ps = dup2(a.post_scale);
    reinterpret_cast<uint4*>(a.mm)[cg] = ldexp_down4(mul4(s1[0], ratio2), a.mean_levels);
    reinterpret_cast<uint4*>(a.mm)[tc + cg] = ldexp_down4(mul4(s2[0], ratio2), a.mean_levels);
    const uint4 sum1 = s1[0], sum2 = s2[0];
    if (swap) {
      reinterpret_cast<uint4*>(a.dbeta)[cg] = sum1;
      reinterpret_cast<uint4*>(a.dgamma)[cg] = add4(mul4(sum2, ps), s3[0]);
    } else {
      reinterpret_cast<uint4*>(a.dbeta)[cg] = mul4(sum1, ps);
      reinterpret_cast<uint4*>(a.dgamma)[cg] = mul4(sum2, ps);
    }
  }
}

// Final forward statistics from a conv-output statistics buffer (written by
// pf16_conv_fwd_bnstats): a balanced tree over the buffer's slots (padded to a
// power of two with empty nodes), each slot a (mean, variance, count) node of
// one epilogue warp, merged by the count-aware parallel-variance rule.  One
// CTA per channel group of 8.
__global__ void __launch_bounds__(kFinalThreads)
    k_bn_fwd_final_slots(const uint8_t* __restrict__ stats, int C, uint16_t eps, uint16_t* mean_out,
                         uint16_t* invstd_out) {
  pdl_wait();
  __shared__ uint4 smu[kFinalThreads], sv[kFinalThreads];
  __shared__ long long sn[kFinalThreads];
  const int cg = blockIdx.x, t = threadIdx.x;
  const uint16_t* smean = reinterpret_cast<const uint16_t*>(stats + bnstat_off_mean());
  const uint16_t* svar = reinterpret_cast<const uint16_t*>(stats + bnstat_off_var(C));
  const int* scnt = reinterpret_cast<const int*>(stats + bnstat_off_cnt(C));
  // slot t's node, loaded before the slot count is known (the buffer holds
  // kBnStatSlots = kFinalThreads slots, so the loads stay inside it)
  const uint4 pm = __ldg(reinterpret_cast<const uint4*>(smean + (long long)t * C) + cg);
  const uint4 pv = __ldg(reinterpret_cast<const uint4*>(svar + (long long)t * C) + cg);
  const long long pn = __ldg(scnt + t);
  const int S = *reinterpret_cast<const int*>(stats);
  int sp2 = 1;
  while (sp2 < S) sp2 *= 2;
  if (sp2 <= kFinalThreads) {
    // one slot per thread and the same strided tree as below: its levels of
    // 32 and more in shared memory, the rest by shuffles in warp 0
    const MV node = t < S ? MV{pm, pv, pn} : MV{zero4(), zero4(), 0ll};
    smu[t] = node.mu;
    sv[t] = node.v;
    sn[t] = node.n;
    __syncthreads();
    for (int half = sp2 / 2; half >= 32; half /= 2) {
      if (t < half) {
        const MV r = mv_merge(MV{smu[t], sv[t], sn[t]}, MV{smu[t + half], sv[t + half], sn[t + half]});
        smu[t] = r.mu;
        sv[t] = r.v;
        sn[t] = r.n;
      }
      __syncthreads();
    }
    if (t >= 32) return;
    MV r{smu[t], sv[t], sn[t]};
    for (int half = sp2 / 2 < 16 ? sp2 / 2 : 16; half >= 1; half /= 2) {
      const MV o{shfl_down4(r.mu, half), shfl_down4(r.v, half), __shfl_down_sync(0xffffffffu, r.n, half)};
      if (t < half) r = mv_merge(r, o);
    }
    if (t == 0) {
      const uint4 ve = add4(r.v, make_uint4(dup2(eps), dup2(eps), dup2(eps), dup2(eps)));
      uint4 is;
      const __half2* hv = reinterpret_cast<const __half2*>(&ve);
      __half2* hi = reinterpret_cast<__half2*>(&is);
#pragma unroll
      for (int j = 0; j < 4; ++j) hi[j] = h2rsqrt(hv[j]);
      reinterpret_cast<uint4*>(mean_out)[cg] = r.mu;
      reinterpret_cast<uint4*>(invstd_out)[cg] = is;
    }
    return;
  }
  const int nthr = sp2 < kFinalThreads ? sp2 : kFinalThreads;
  const int seg = sp2 / nthr;
  if (t < nthr) {
    MV st[12];
    unsigned cnt = 0;
    for (int i = 0; i < seg; ++i) {
      const int b = t * seg + i;
      const bool ok = b < S;
      MV node{ok ? __ldg(reinterpret_cast<const uint4*>(smean + (long long)b * C) + cg) : zero4(),
              ok ? __ldg(reinterpret_cast<const uint4*>(svar + (long long)b * C) + cg) : zero4(),
              ok ? (long long)__ldg(scnt + b) : 0ll};
#pragma unroll
      for (int l = 0; l < 12; ++l) {
        if (cnt & (1u << l)) {
          node = mv_merge(st[l], node);
        } else {
          st[l] = node;
          break;
        }
      }
      ++cnt;
    }
    const int lv = 31 - __clz(seg);
    MV res = st[0];
#pragma unroll
    for (int l = 0; l < 12; ++l)
      if (l == lv) res = st[l];
    smu[t] = res.mu;
    sv[t] = res.v;
    sn[t] = res.n;
  }
  __syncthreads();
  for (int half = nthr / 2; half >= 1; half /= 2) {
    if (t < half) {
      const MV r = mv_merge(MV{smu[t], sv[t], sn[t]}, MV{smu[t + half], sv[t + half], sn[t + half]});
      smu[t] = r.mu;
      sv[t] = r.v;
      sn[t] = r.n;
    }
    __syncthreads();
  }
  if (t == 0) {
    const uint4 ve = add4(sv[0], make_uint4(dup2(eps), dup2(eps), dup2(eps), dup2(eps)));
    uint4 is;
    const __half2* hv = reinterpret_cast<const __half2*>(&ve);
    __half2* hi = reinterpret_cast<__half2*>(&is);
#pragma unroll
    for (int j = 0; j < 4; ++j) hi[j] = h2rsqrt(hv[j]);
    reinterpret_cast<uint4*>(mean_out)[cg] = smu[0];
    reinterpret_cast<uint4*>(invstd_out)[cg] = is;
  }
}

// Backward statistics from a dgrad statistics buffer (pf16_conv_dgrad_bnstats):
// the slots hold pairwise sums of dy' and dy' * xhat; a pairwise tree over
// the slots (padded to a power of two with zeros) closes the sums, then, as
// k_bn_bwd_final, dbeta / dgamma = rn(sum * post_scale) and the means
// rn(rn(sum * rn(2^L/R)) * 2^-L), L = ceil(log2 R).  One CTA per channel
// group of 8.
__global__ void __launch_bounds__(kFinalThreads)
    k_bn_bwd_final_slots(const uint8_t* __restrict__ stats, int C, int mean_levels, uint16_t ratio,
                         uint16_t post_scale, uint16_t* mm, uint16_t* dgamma, uint16_t* dbeta) {
  pdl_wait();
  __shared__ uint4 s1[kFinalThreads], s2[kFinalThreads];
  const int tc = C / 8, cg = blockIdx.x, t = threadIdx.x;
  const uint16_t* sd = reinterpret_cast<const uint16_t*>(stats + bnstat_off_mean());
  const uint16_t* sp = reinterpret_cast<const uint16_t*>(stats + bnstat_off_var(C));
  // slot t's sums, loaded before the slot count is known (as the forward's final)
  const uint4 p1 = __ldg(reinterpret_cast<const uint4*>(sd + (long long)t * C) + cg);
  const uint4 p2 = __ldg(reinterpret_cast<const uint4*>(sp + (long long)t * C) + cg);
  const int S = reinterpret_cast<const int*>(stats)[0];
  int sp2 = 1;
  while (sp2 < S) sp2 *= 2;
  if (sp2 <= kFinalThreads) {
    // one slot per thread and the same strided tree as below: its levels of
    // 32 and more in shared memory, the rest by shuffles in warp 0
    s1[t] = t < S ? p1 : zero4();
    s2[t] = t < S ? p2 : zero4();
    __syncthreads();
    for (int half = sp2 / 2; half >= 32; half /= 2) {
      if (t < half) {
        s1[t] = add4(s1[t], s1[t + half]);
        s2[t] = add4(s2[t], s2[t + half]);
      }
      __syncthreads();
    }
    if (t >= 32) return;
    uint4 a1 = s1[t], a2 = s2[t];
    for (int half = sp2 / 2 < 16 ? sp2 / 2 : 16; half >= 1; half /= 2) {
      const uint4 o1 = shfl_down4(a1, half), o2 = shfl_down4(a2, half);
      if (t < half) {
        a1 = add4(a1, o1);
        a2 = add4(a2, o2);
      }
    }
    if (t == 0) {
      const uint32_t ratio2 = dup2(ratio), ps = dup2(post_scale);
      reinterpret_cast<uint4*>(mm)[cg] = ldexp_down4(mul4(a1, ratio2), mean_levels);
      reinterpret_cast<uint4*>(mm)[tc + cg] = ldexp_down4(mul4(a2, ratio2), mean_levels);
      reinterpret_cast<uint4*>(dbeta)[cg] = mul4(a1, ps);
      reinterpret_cast<uint4*>(dgamma)[cg] = mul4(a2, ps);
    }
    return;
  }
  const int nthr = sp2 < kFinalThreads ? sp2 : kFinalThreads;
  const int seg = sp2 / nthr;
  if (t < nthr) {
    Tree4<12, false> t1, t2;
    for (int i = 0; i < seg; ++i) {
      const int b = t * seg + i;
      const bool ok = b < S;
      t1.push(ok ? __ldg(reinterpret_cast<const uint4*>(sd + (long long)b * C) + cg) : zero4());
      t2.push(ok ? __ldg(reinterpret_cast<const uint4*>(sp + (long long)b * C) + cg) : zero4());
    }
    const int lv = 31 - __clz(seg);
    s1[t] = t1.finish(lv);
    s2[t] = t2.finish(lv);
  }
  __syncthreads();
  for (int half = nthr / 2; half >= 1; half /= 2) {
    if (t < half) {
      s1[t] = add4(s1[t], s1[t + half]);
      s2[t] = add4(s2[t], s2[t + half]);
    }
    __syncthreads();
  }
  if (t == 0) {
    const uint32_t ratio2 = dup2(ratio), ps = dup2(post_scale);
    reinterpret_cast<uint4*>(mm)[cg] = ldexp_down4(mul4(s1[0], ratio2), mean_levels);
    reinterpret_cast<uint4*>(mm)[tc + cg] = ldexp_down4(mul4(s2[0], ratio2), mean_levels);
    reinterpret_cast<uint4*>(dbeta)[cg] = mul4(s1[0], ps);
    reinterpret_cast<uint4*>(dgamma)[cg] = mul4(s2[0], ps);
  }
}

constexpr int kApplyRows = 8;  // rows per thread per CTA in the apply passes
// rows whose loads are issued together: all eight in the backward apply (a
// shorter dependency chain for the small late-stage tensors: 10-30% faster
// there), four in the forward's (which measured slower with eight)
constexpr int kApplyBatch = 8;
constexpr int kApplyBatchFwd = 4;

__global__ void __launch_bounds__(256)
    k_bn_apply(const uint16_t* __restrict__ x, const uint16_t* __restrict__ gamma,
               const uint16_t* __restrict__ beta, const uint16_t* __restrict__ mean,
               const uint16_t* __restrict__ invstd, const uint16_t* __restrict__ residual,
               uint16_t* __restrict__ y, uint8_t* __restrict__ mask, int R, int C, int rpb,
               uint16_t post_scale, int relu, int swap) {
  pdl_wait();
  const int tc = C / 8;
  const int t = threadIdx.x;
  if (t >= tc * rpb) return;
  const int cg = t % tc, rg = t / tc;
  const uint32_t ps = dup2(post_scale);
  const uint4 mu = __ldg(reinterpret_cast<const uint4*>(mean) + cg);
  const uint4 is = __ldg(reinterpret_cast<const uint4*>(invstd) + cg);
  const uint4 ga = __ldg(reinterpret_cast<const uint4*>(gamma) + cg);
  const uint4 be = __ldg(reinterpret_cast<const uint4*>(beta) + cg);
  const long long row0 = (long long)blockIdx.x * rpb * kApplyRows;
#pragma unroll
  for (int h = 0; h < kApplyRows; h += kApplyBatchFwd) {
    uint4 xv[kApplyBatchFwd], rv[kApplyBatchFwd];
#pragma unroll
    for (int i = 0; i < kApplyBatchFwd; ++i) {
      const long long r = row0 + rg + (long long)(h + i) * rpb;
      const long long off = r * tc + cg;
      xv[i] = r < R ? __ldg(reinterpret_cast<const uint4*>(x) + off) : zero4();
      rv[i] = (r < R && residual) ? __ldg(reinterpret_cast<const uint4*>(residual) + off) : zero4();
    }
#pragma unroll
    for (int i = 0; i < kApplyBatchFwd; ++i) {
      const long long r = row0 + rg + (long long)(h + i) * rpb;
      if (r >= R) break;
      const uint4 xh = mul4v(sub4(xv[i], mu), is);      // Eq. 1
      uint4 z;
      if (swap)  // Sec. 4.1: gamma * (s * xhat + residual) + beta
        z = add4(mul4v(ga, add4(mul4(xh, ps), rv[i])), be);
      else {
        z = mul4(add4(mul4v(ga, xh), be), ps);          // Eq. 2, then x post_scale
        if (residual) z = add4(z, rv[i]);
      }
      if (relu) {
        uint32_t bits;
        z = relu_bits(z, bits);
        if (mask) mask[r * tc + cg] = (uint8_t)bits;
      }
      reinterpret_cast<uint4*>(y)[r * tc + cg] = z;
    }
  }
}

template <int RELU>
__global__ void __launch_bounds__(256)
    k_bn_bwd_apply(const uint16_t* __restrict__ x, const uint16_t* __restrict__ gamma,
                   const uint16_t* __restrict__ mean, const uint16_t* __restrict__ invstd,
                   const uint16_t* __restrict__ dy, const uint16_t* __restrict__ y_saved,
                   const uint8_t* __restrict__ mask, const uint16_t* __restrict__ mm,
                   uint16_t* __restrict__ dx, uint16_t* __restrict__ dres, int R, int C, int rpb,
                   uint16_t post_scale, int swap) {
  pdl_wait();
  const int tc = C / 8;
  const int t = threadIdx.x;
  if (t >= tc * rpb) return;
  const int cg = t % tc, rg = t / tc;
  const uint32_t ps = dup2(post_scale);
  const uint4 mu = __ldg(reinterpret_cast<const uint4*>(mean) + cg);
  const uint4 is = __ldg(reinterpret_cast<const uint4*>(invstd) + cg);
  const uint4 ga = __ldg(reinterpret_cast<const uint4*>(gamma) + cg);
  const uint4 m1 = __ldg(reinterpret_cast<const uint4*>(mm) + cg);
  const uint4 m2 = __ldg(reinterpret_cast<const uint4*>(mm) + tc + cg);
  const uint4 k = mul4v(mul4(ga, ps), is);  // s * gamma * invstd
  const long long row0 = (long long)blockIdx.x * rpb * kApplyRows;
#pragma unroll
  for (int h = 0; h < kApplyRows; h += kApplyBatch) {  // all of a thread's rows in flight at once
    uint4 xs[kApplyBatch], ds[kApplyBatch], ys[kApplyBatch];
    uint32_t mb[kApplyBatch];
#pragma unroll
    for (int i = 0; i < kApplyBatch; ++i) {
      const long long r = row0 + rg + (long long)(h + i) * rpb;
      const long long off = r * tc + cg;
      const bool ok = r < R;
      ds[i] = ok ? __ldg(reinterpret_cast<const uint4*>(dy) + off) : zero4();
      xs[i] = ok ? __ldg(reinterpret_cast<const uint4*>(x) + off) : zero4();
      if (RELU == BN_RELU_SAVED) ys[i] = ok ? __ldg(reinterpret_cast<const uint4*>(y_saved) + off) : zero4();
      if (RELU == BN_RELU_BITS) mb[i] = ok ? (uint32_t)__ldg(mask + off) : 0u;
    }
#pragma unroll
    for (int i = 0; i < kApplyBatch; ++i) {
      const long long r = row0 + rg + (long long)(h + i) * rpb;
      if (r >= R) break;
      uint4 d = ds[i];
      if (RELU == BN_RELU_SAVED) d = and4(d, relu_mask4(ys[i]));
      if (RELU == BN_RELU_BITS) d = and4(d, bits_mask4(mb[i]));
      const uint4 xh = mul4v(sub4(xs[i], mu), is);
      const uint4 tt = sub4(sub4(d, m1), mul4v(xh, m2));  // dy' - mean(dy') - xhat*mean(dy'*xhat)
      const long long off = r * tc + cg;
      reinterpret_cast<uint4*>(dx)[off] = mul4v(k, tt);
      if (dres) reinterpret_cast<uint4*>(dres)[off] = swap ? mul4v(ga, d) : d;  // swap: gamma * dy' 
    }
  }
}

unsigned grid_for(long long work, int per_block, int cap) {
  long long b = (work + per_block - 1) / per_block;
  if (b < 1) b = 1;
  if (b > cap) b = cap;
  return (unsigned)b;
}

}  // namespace

static BnPlan bn_stat_plan(long long chunks, int ctas_per_sm) {
  BnPlan p;
  long long grid = (long long)kGb300Sms * ctas_per_sm;  // the fixed statistics grid
  if (chunks > grid * kStatMaxChunks) grid = (chunks + kStatMaxChunks - 1) / kStatMaxChunks;
  if (grid > chunks) grid = chunks;
  p.blocks = (int)grid;
  p.chunks_per_cta = (int)((chunks + grid - 1) / grid);
  int p2 = 1;
  while (p2 < p.blocks) p2 *= 2;
  p.blocks_pow2 = p2;
  return p;
}

void bn_plan(int R, int C, BnLaunch* b) {
  b->R = R;
  b->C = C;
  const BnGeom g = bn_geom(C);
  b->chunk_rows = g.rpb * kStatRowsT;
  const long long chunks = ((long long)R + b->chunk_rows - 1) / b->chunk_rows;
  b->fwd = bn_stat_plan(chunks, kFwdCtasPerSm);
  b->bwd = bn_stat_plan(chunks, kBwdCtasPerSm);
}

// [ws1: blocks*C] [ws2: blocks*C] [mm: 2*C]
size_t bn_ws_bytes(const BnLaunch& b) {
  const size_t blocks = (size_t)(b.fwd.blocks > b.bwd.blocks ? b.fwd.blocks : b.bwd.blocks);
  // [ws1][ws2][mm] (+ the swap variant's second pass: [ws3][ws4])
  return 256 + (b.swap ? 4 : 2) * blocks * b.C * sizeof(uint16_t) + (size_t)2 * b.C * sizeof(uint16_t) + 256;
}

static uint16_t f16_bits_host(float f) {
  __half h = __float2half_rn(f);
  return *reinterpret_cast<uint16_t*>(&h);
}

static BnStatArgs bn_args(const BnLaunch& b, const BnPlan& p, uint16_t* ws) {
  BnStatArgs a;
  memset(&a, 0, sizeof(a));
  a.R = b.R;
  a.C = b.C;
  a.blocks = p.blocks;
  a.blocks_pow2 = p.blocks_pow2;
  a.chunk_levels = ceil_log2(p.chunks_per_cta);
  // backward means: sum * rn(2^L / R) * 2^-L, L = ceil(log2 R)
  a.mean_levels = ceil_log2(b.R);
  a.ratio = f16_bits_host((float)(ldexp(1.0, a.mean_levels) / (double)b.R));
  a.eps = b.eps;
  a.post_scale = b.post_scale;
  a.status = b.status;
  a.wait_limit_ns = 4000000000ull;
  a.ws1 = ws;
  a.ws2 = a.ws1 + (size_t)p.blocks * b.C;
  a.mm = a.ws2 + (size_t)p.blocks * b.C;
  return a;
}

// Opt a statistics kernel into its dynamic shared memory once per device.
template <typename K>
static cudaError_t stat_smem_attr(K kernel, int bytes, bool* done) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!done[dev]) {
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e != cudaSuccess) return e;
    done[dev] = true;
  }
  return cudaSuccess;
}

cudaError_t launch_bn_fwd(const BnLaunch& b, const uint16_t* x, const uint16_t* gamma,
                          const uint16_t* beta, const uint16_t* residual, uint16_t* y,
                          uint8_t* relu_mask, uint16_t* mean, uint16_t* invstd, uint16_t* ws,
                          cudaStream_t s) {
  static bool attr[64] = {false};
  cudaError_t e = stat_smem_attr(k_bn_fwd_stats, stat_smem_bytes(1), attr);
  if (e != cudaSuccess) return e;
  BnStatArgs a = bn_args(b, b.fwd, ws);
  a.x = x;
  a.mean_out = mean;
  a.invstd_out = invstd;
  const BnGeom g = bn_geom(b.C);
  launch_pdl(k_bn_fwd_stats, dim3(b.fwd.blocks), dim3(g.threads + 32), stat_smem_bytes(1), s, a);
  launch_pdl(k_bn_fwd_final, dim3(b.C / 8), dim3(kFinalThreads), 0, s, a, (long long)b.chunk_rows);
  if (!y) return counted_launches(2);  // statistics only
  const int rows = g.rpb * kApplyRows;
  launch_pdl(k_bn_apply, dim3((unsigned)((b.R + rows - 1) / rows)), dim3(g.threads), 0, s, 
      x, gamma, beta, mean, invstd, residual, y, b.relu ? relu_mask : nullptr, b.R, b.C, g.rpb,
      b.post_scale, b.relu, b.swap);
  return counted_launches(3);
}

cudaError_t launch_bn_fwd_given_stats(const BnLaunch& b, const uint8_t* conv_stats, const uint16_t* x,
                                      const uint16_t* gamma, const uint16_t* beta,
                                      const uint16_t* residual, uint16_t* y, uint8_t* relu_mask,
                                      uint16_t* mean, uint16_t* invstd, cudaStream_t s) {
  launch_pdl(k_bn_fwd_final_slots, dim3(b.C / 8), dim3(kFinalThreads), 0, s, conv_stats, b.C, b.eps, mean, invstd);
  if (!y) return counted_launches(1);  // statistics only
  const BnGeom g = bn_geom(b.C);
  const int rows = g.rpb * kApplyRows;
  launch_pdl(k_bn_apply, dim3((unsigned)((b.R + rows - 1) / rows)), dim3(g.threads), 0, s, 
      x, gamma, beta, mean, invstd, residual, y, b.relu ? relu_mask : nullptr, b.R, b.C, g.rpb,
      b.post_scale, b.relu, b.swap);
  return counted_launches(2);
}

// One backward statistics pass of mode RELU (XRAW: the second tree sums dy' * x).
template <int RELU, bool XRAW>
static cudaError_t bwd_stats_pass(const BnStatArgs& a, const BnLaunch& b, cudaStream_t s) {
  static bool attr[64] = {false};
  const int smem = stat_smem_bytes(2);
  cudaError_t e = stat_smem_attr(k_bn_bwd_stats<RELU, XRAW>, smem, attr);
  if (e != cudaSuccess) return e;
  const BnGeom g = bn_geom(b.C);
  launch_pdl(k_bn_bwd_stats<RELU, XRAW>, dim3(b.bwd.blocks), dim3((unsigned)(g.threads + 32)), smem, s, a);
  return cudaSuccess;
}
template <bool XRAW>
static cudaError_t bwd_stats_mode(int mode, const BnStatArgs& a, const BnLaunch& b, cudaStream_t s) {
  switch (mode) {
    case BN_NO_RELU: return bwd_stats_pass<BN_NO_RELU, XRAW>(a, b, s);
    case BN_RELU_SAVED: return bwd_stats_pass<BN_RELU_SAVED, XRAW>(a, b, s);
    default: return bwd_stats_pass<BN_RELU_BITS, XRAW>(a, b, s);
  }
}

cudaError_t launch_bn_bwd(const BnLaunch& b, const uint16_t* x, const uint16_t* gamma,
                          const uint16_t* mean, const uint16_t* invstd, const uint16_t* dy,
                          const uint16_t* y_saved, const uint8_t* relu_mask, uint16_t* dx,
                          uint16_t* dgamma, uint16_t* dbeta, uint16_t* dres, uint16_t* ws,
                          cudaStream_t s, const uint8_t* dgrad_stats, const uint16_t* residual) {
  BnStatArgs a = bn_args(b, b.bwd, ws);
  a.x = x;
  a.dy = dy;
  a.y_saved = y_saved;
  a.mask_in = relu_mask;
  a.mean_in = mean;
  a.invstd_in = invstd;
  a.dgamma = dgamma;
  a.dbeta = dbeta;
  const BnGeom g = bn_geom(b.C);
  const int mode = !b.relu ? BN_NO_RELU : (relu_mask ? BN_RELU_BITS : BN_RELU_SAVED);
  const int rows = g.rpb * kApplyRows;
  const unsigned apply_blocks = (unsigned)((b.R + rows - 1) / rows);
  cudaError_t e = cudaSuccess;
  int launches = 3;
  if (dgrad_stats) {
    // statistics from the producing data gradient's epilogue
    launch_pdl(k_bn_bwd_final_slots, dim3(b.C / 8), dim3(kFinalThreads), 0, s, dgrad_stats, b.C, a.mean_levels,
               a.ratio, b.post_scale, a.mm, dgamma, dbeta);
    launches = 2;
  } else {
    if ((e = bwd_stats_mode<false>(mode, a, b, s)) != cudaSuccess) return e;
    if (b.swap) {
      // the swap variant's dgamma also needs sum dy' * residual: the same pass over
      // (residual, dy) with the raw second tree, into its own per-CTA buffers
      BnStatArgs a2 = a;
      a2.x = residual;
      a2.ws1 = a.mm + 2 * (size_t)b.C;
      a2.ws2 = a2.ws1 + (size_t)b.bwd.blocks * b.C;
      a.ws4 = a2.ws2;
      if ((e = bwd_stats_mode<true>(mode, a2, b, s)) != cudaSuccess) return e;
      ++launches;
    }
    launch_pdl(k_bn_bwd_final, dim3(b.C / 8), dim3(kFinalThreads), 0, s, a);
  }
  switch (mode) {
    case BN_NO_RELU:
      launch_pdl(k_bn_bwd_apply<BN_NO_RELU>, dim3(apply_blocks), dim3(g.threads), 0, s, 
          x, gamma, mean, invstd, dy, nullptr, nullptr, a.mm, dx, dres, b.R, b.C, g.rpb, b.post_scale, b.swap);
      break;
    case BN_RELU_SAVED:
      launch_pdl(k_bn_bwd_apply<BN_RELU_SAVED>, dim3(apply_blocks), dim3(g.threads), 0, s, 
          x, gamma, mean, invstd, dy, y_saved, nullptr, a.mm, dx, dres, b.R, b.C, g.rpb, b.post_scale, b.swap);
      break;
    default:
      launch_pdl(k_bn_bwd_apply<BN_RELU_BITS>, dim3(apply_blocks), dim3(g.threads), 0, s, 
          x, gamma, mean, invstd, dy, nullptr, relu_mask, a.mm, dx, dres, b.R, b.C, g.rpb, b.post_scale, b.swap);
      break;
  }
  return counted_launches(launches);
}

// ============================================================================
// Max pooling 3x3 / stride 2 / pad 1 and its backward (first-max rule).
// ============================================================================
// Forward, one CTA per output row (n, p); with `codes` it also records, per
// output element, the position r*3+s of the window's first maximum (r then s
// order, padding excluded).
__global__ void __launch_bounds__(256)
    k_maxpool_fwd(const uint16_t* __restrict__ x, uint16_t* __restrict__ y, uint8_t* __restrict__ codes,
                  int N, int H, int W, int C, int P, int Q) {
  pdl_wait();
  const int tc = C / 8;
  const int n = blockIdx.x / P, p = blockIdx.x - n * P;
  const long long orow = (long long)blockIdx.x * Q * tc;  // first output vector of the row
  for (int i = threadIdx.x; i < Q * tc; i += blockDim.x) {
    const int q = i / tc, cg = i - q * tc;
    float m[8];
    uint32_t code[2] = {0xFFFFFFFFu, 0xFFFFFFFFu};
#pragma unroll
    for (int e = 0; e < 8; ++e) m[e] = -INFINITY;
    for (int r = 0; r < 3; ++r) {
      const int h = 2 * p + r - 1;
      if (h < 0 || h >= H) continue;
      const uint4* xrow = reinterpret_cast<const uint4*>(x + ((long long)n * H + h) * W * C);
      for (int s = 0; s < 3; ++s) {
        const int w = 2 * q + s - 1;
        if (w < 0 || w >= W) continue;
        const uint4 v = __ldg(xrow + w * tc + cg);
        const __half* hv = reinterpret_cast<const __half*>(&v);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float f = __half2float(hv[e]);
          if (f > m[e]) {
            m[e] = f;
            const int sh = (e & 3) * 8;
            code[e >> 2] = (code[e >> 2] & ~(0xFFu << sh)) | ((uint32_t)(r * 3 + s) << sh);
          }
        }
      }
    }
    uint4 out;
    __half* ho = reinterpret_cast<__half*>(&out);
#pragma unroll
    for (int e = 0; e < 8; ++e) ho[e] = __float2half_rn(m[e]);  // exact: m is a binary16 value
    reinterpret_cast<uint4*>(y)[orow + i] = out;
    if (codes) reinterpret_cast<uint2*>(codes)[orow + i] = make_uint2(code[0], code[1]);
  }
}

__device__ __forceinline__ uint32_t heq2_mask(uint32_t a, uint32_t b) {  // 0xFFFF per half where a == b
  uint32_t d;
  asm("set.eq.u32.f16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

// Backward from the recorded positions.  Input cells (2i + a, 2j + b),
// a, b in {0, 1}, are covered exactly by the windows p in {i, i+1}, q in
// {j, j+1} (cell row 2i only by p = i, cell column 2j only by q = j), so one
// thread owns that 2x2 block of cells for one group of 8 channels: it loads
// the four windows' positions and gradients once, then every cell sums, in
// window order (p, then q), the gradients of the windows whose first maximum
// it is.  One CTA per block row (n, i).
__global__ void __launch_bounds__(512)
    k_maxpool_bwd_codes(const uint8_t* __restrict__ codes, const uint16_t* __restrict__ dy,
                        uint16_t* __restrict__ dx, int N, int H, int W, int C, int P, int Q) {
  pdl_wait();
  const int tc = C / 8;
  const int HB = (H + 1) / 2, WB = (W + 1) / 2;
  const int n = blockIdx.x / HB, i = blockIdx.x - n * HB;
  for (int t = threadIdx.x; t < WB * tc; t += blockDim.x) {
    const int j = t / tc, cg = t - j * tc;
    uint2 cd[2][2];
    uint4 g[2][2];
#pragma unroll
    for (int a = 0; a < 2; ++a)
#pragma unroll
      for (int b = 0; b < 2; ++b) {
        const int p = i + a, q = j + b;
        const bool ok = p < P && q < Q;
        const long long oi = (((long long)n * P + p) * Q + q) * tc + cg;
        cd[a][b] = ok ? __ldg(reinterpret_cast<const uint2*>(codes) + oi) : make_uint2(~0u, ~0u);
        g[a][b] = ok ? __ldg(reinterpret_cast<const uint4*>(dy) + oi) : make_uint4(0, 0, 0, 0);
      }
    // each window's positions widened to one 16-bit lane per channel (word k:
    // channels 2k, 2k + 1), compared as binary16 bit patterns: 0..8 and 0xFF
    // are zero or subnormal, so f16x2 equality is equality of the codes
    uint32_t cw16[2][2][4];
#pragma unroll
    for (int a = 0; a < 2; ++a)
#pragma unroll
      for (int b = 0; b < 2; ++b)
#pragma unroll
        for (int k = 0; k < 4; ++k)
          cw16[a][b][k] = __byte_perm(k < 2 ? cd[a][b].x : cd[a][b].y, 0u, (k & 1) ? 0x4342 : 0x4140);
#pragma unroll
    for (int ch = 0; ch < 2; ++ch) {
      const int h = 2 * i + ch;
      if (h >= H) break;
#pragma unroll
      for (int cw = 0; cw < 2; ++cw) {
        const int w = 2 * j + cw;
        if (w >= W) break;
        uint32_t acc[4] = {0, 0, 0, 0};
#pragma unroll
        for (int a = 0; a < 2; ++a) {
          if (a > ch) break;  // cell row 2i lies in window row i only
#pragma unroll
          for (int b = 0; b < 2; ++b) {
            if (b > cw) break;
            // the cell's position in window (i + a, j + b): row ch - 2a + 1,
            // column cw - 2b + 1, in both halves
            const uint32_t mine = (uint32_t)((ch - 2 * a + 1) * 3 + (cw - 2 * b + 1)) * 0x00010001u;
            const uint32_t* gw = reinterpret_cast<const uint32_t*>(&g[a][b]);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const uint32_t sel = heq2_mask(cw16[a][b][k], mine);
              if (sel) acc[k] = hadd2_rn(acc[k], gw[k] & sel);
            }
          }
        }
        reinterpret_cast<uint4*>(dx)[(((long long)n * H + h) * W + w) * tc + cg] =
            make_uint4(acc[0], acc[1], acc[2], acc[3]);
      }
    }
  }
}

// Backward.  A CTA owns output-window rows [p0, p0 + kPoolTP) of one image
// and one group of 8 channels, i.e. input rows [2 p0, 2 p0 + 2 kPoolTP).  It
// stages input rows 2 p0 - 1 .. 2 p0 + 2 kPoolTP + 1 in shared memory, finds
// each window's first maximum once (code r*3+s per channel, 0xFF if the
// window has no valid cell), then every owned cell sums, in window order, the
// gradients of the windows whose maximum it holds.
constexpr int kPoolTP = 4;

__global__ void __launch_bounds__(256)
    k_maxpool_bwd(const uint16_t* __restrict__ x, const uint16_t* __restrict__ dy,
                  uint16_t* __restrict__ dx, int N, int H, int W, int C, int P, int Q) {
  pdl_wait();
  extern __shared__ uint4 band[];  // [2*kPoolTP + 3][W] cells of 8 channels
  const int tc = C / 8;
  const int bands = (P + kPoolTP - 1) / kPoolTP;
  const int cg = blockIdx.x % tc;
  const int rest = blockIdx.x / tc;
  const int pb = rest % bands, n = rest / bands;
  const int p0 = pb * kPoolTP;
  const int h0 = 2 * p0 - 1;  // input row held in band row 0
  constexpr int BR = 2 * kPoolTP + 3;
  uint8_t* codes = reinterpret_cast<uint8_t*>(band + BR * W);  // [kPoolTP + 1][Q][8]
  for (int i = threadIdx.x; i < BR * W; i += blockDim.x) {
    const int br = i / W, w = i - br * W;
    const int h = h0 + br;
    band[i] = (h >= 0 && h < H) ? __ldg(reinterpret_cast<const uint4*>(x + (((long long)n * H + h) * W + w) * C) + cg)
                                : make_uint4(0, 0, 0, 0);
  }
  __syncthreads();
  for (int i = threadIdx.x; i < (kPoolTP + 1) * Q; i += blockDim.x) {
    const int pp = i / Q, q = i - pp * Q;
    const int p = p0 + pp;
    float m[8];
    uint8_t code[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      m[e] = -INFINITY;
      code[e] = 0xFF;
    }
    if (p < P) {
      for (int r = 0; r < 3; ++r) {
        const int h = 2 * p + r - 1;
        if (h < 0 || h >= H) continue;
        for (int c = 0; c < 3; ++c) {
          const int w = 2 * q + c - 1;
          if (w < 0 || w >= W) continue;
          const uint4 v = band[(h - h0) * W + w];
          const __half* hv = reinterpret_cast<const __half*>(&v);
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const float f = __half2float(hv[e]);
            if (f > m[e]) {
              m[e] = f;
              code[e] = (uint8_t)(r * 3 + c);
            }
          }
        }
      }
    }
#pragma unroll
    for (int e = 0; e < 8; ++e) codes[i * 8 + e] = code[e];
  }
  __syncthreads();
  for (int i = threadIdx.x; i < 2 * kPoolTP * W; i += blockDim.x) {
    const int hh = i / W, w = i - hh * W;
    const int h = 2 * p0 + hh;
    if (h >= H) continue;
    uint32_t acc[4] = {0, 0, 0, 0};
    const int p_lo = h / 2, p_hi = (h + 1) / 2;  // windows covering row h
    for (int p = p_lo; p <= p_hi; ++p) {
      if (p >= P || h < 2 * p - 1 || h > 2 * p + 1) continue;
      const int pp = p - p0;  // 0 .. kPoolTP
      for (int q = w / 2; q <= (w + 1) / 2; ++q) {
        if (q >= Q || w < 2 * q - 1 || w > 2 * q + 1) continue;
        const uint8_t* cd = codes + (pp * Q + q) * 8;
        const uint8_t mine = (uint8_t)((h - (2 * p - 1)) * 3 + (w - (2 * q - 1)));
        uint32_t sel[4];
        bool any = false;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          sel[j] = (cd[2 * j] == mine ? 0x0000FFFFu : 0u) | (cd[2 * j + 1] == mine ? 0xFFFF0000u : 0u);
          any |= sel[j] != 0;
        }
        if (!any) continue;
        const uint4 g = __ldg(reinterpret_cast<const uint4*>(dy + (((long long)n * P + p) * Q + q) * C) + cg);
        const uint32_t* gw = reinterpret_cast<const uint32_t*>(&g);
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (sel[j]) acc[j] = hadd2_rn(acc[j], gw[j] & sel[j]);
      }
    }
    reinterpret_cast<uint4*>(dx + (((long long)n * H + h) * W + w) * C)[cg] =
        make_uint4(acc[0], acc[1], acc[2], acc[3]);
  }
}

cudaError_t launch_maxpool_fwd(const uint16_t* x, uint16_t* y, uint8_t* codes, int N, int H, int W,
                               int C, cudaStream_t s) {
  const int P = (H - 1) / 2 + 1, Q = (W - 1) / 2 + 1;
  launch_pdl(k_maxpool_fwd, dim3((unsigned)((long long)N * P)), dim3(256), 0, s, x, y, codes, N, H, W, C, P, Q);
  return counted_launches(1);
}

cudaError_t launch_maxpool_bwd_codes(const uint8_t* codes, const uint16_t* dy, uint16_t* dx, int N,
                                     int H, int W, int C, cudaStream_t s) {
  const int P = (H - 1) / 2 + 1, Q = (W - 1) / 2 + 1;
  // one thread per 2x2 cell block of a block row, where that fits in 512 threads
  const long long per_row = (long long)((W + 1) / 2) * (C / 8);
  const int threads = per_row >= 512 ? 512 : (int)((per_row + 31) / 32 * 32);
  launch_pdl(k_maxpool_bwd_codes, dim3((unsigned)((long long)N * ((H + 1) / 2))), dim3(threads), 0, s, codes, dy, dx, N, H,
                                                                                     W, C, P, Q);
  return counted_launches(1);
}

cudaError_t launch_maxpool_bwd(const uint16_t* x, const uint16_t* dy, uint16_t* dx, int N, int H,
                               int W, int C, cudaStream_t s) {
  const int P = (H - 1) / 2 + 1, Q = (W - 1) / 2 + 1;
  const int bands = (P + kPoolTP - 1) / kPoolTP;
  const size_t shm = (size_t)(2 * kPoolTP + 3) * W * sizeof(uint4) + (size_t)(kPoolTP + 1) * Q * 8;
  if (shm > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(k_maxpool_bwd, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)shm);
    if (e != cudaSuccess) return e;
  }
  launch_pdl(k_maxpool_bwd, dim3((unsigned)((long long)N * bands * (C / 8))), dim3(256), shm, s, x, dy, dx, N, H, W, C, P, Q);
  return counted_launches(1);
}

// ============================================================================
// The stem's BatchNorm, ReLU and 3x3 / stride 2 / pad 1 max pooling in one
// pass (pf16_bn_relu_maxpool_fwd): y = ReLU(BN(x)) is never stored.  A CTA
// owns kBpT output rows p0 .. p0 + kBpT - 1 of one image, i.e. input rows
// 2 p0 .. 2 p0 + 2 kBpT - 1, whose ReLU bits it writes.  It computes y for
// input rows 2 p0 - 1 .. 2 p0 + 2 kBpT - 1 into shared memory (row 2 p0 - 1
// belongs to the previous CTA and is computed twice) with k_bn_apply's op
// sequence, then takes each window's first maximum (rows then columns, as
// k_maxpool_fwd) from there.  After the ReLU every value is +0 or positive,
// where FP16 order is the order of the bit patterns, so the window scan
// starts from its first valid cell and replaces the maximum where a cell is
// strictly greater (set.gt on f16x2, exact for these values): the pooled
// output and positions are those of k_maxpool_fwd on y, bit for bit.
// ============================================================================
constexpr int kBpT = 2;

__device__ __forceinline__ uint32_t hgt2_mask(uint32_t a, uint32_t b) {  // 0xFFFF per half where a > b
  uint32_t d;
  asm("set.gt.u32.f16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

// take cell value v (position rs) into the window's running maximum m / codes
__device__ __forceinline__ void pool_take(uint4& m, uint32_t (&code)[2], const uint4& v, uint32_t rs) {
  const uint32_t rsr = rs * 0x01010101u;
  uint32_t* mw = &m.x;
  const uint32_t* vw = &v.x;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const uint32_t gt = hgt2_mask(vw[k], mw[k]);
    mw[k] = (vw[k] & gt) | (mw[k] & ~gt);
    // the position bytes of halves 2k, 2k+1: bytes 2(k&1), 2(k&1)+1 of code word k/2
    const uint32_t bm = __byte_perm(gt, 0u, 0x4420) << (16 * (k & 1));
    code[k >> 1] = (code[k >> 1] & ~bm) | (rsr & bm);
  }
}

__global__ void __launch_bounds__(256)
    k_bn_relu_pool_fwd(const uint16_t* __restrict__ x, const uint16_t* __restrict__ gamma,
                       const uint16_t* __restrict__ beta, const uint16_t* __restrict__ mean,
                       const uint16_t* __restrict__ invstd, uint16_t post_scale, uint16_t* __restrict__ pooled,
                       uint8_t* __restrict__ codes, uint8_t* __restrict__ mask, int N, int H, int W, int C, int P,
                       int Q) {
  pdl_wait();
  extern __shared__ uint4 zs[];  // [2 kBpT + 1][W][C / 8]: y of the staged input rows
  const int tc = C / 8;
  const int nb = (P + kBpT - 1) / kBpT;
  const int n = blockIdx.x / nb, p0 = (blockIdx.x - n * nb) * kBpT;
  const uint32_t ps = dup2(post_scale);
  // blockDim is a multiple of tc: a thread keeps one channel group throughout
  // and steps over cells (then windows) by cstep
  const int cg = threadIdx.x % tc, c0 = threadIdx.x / tc, cstep = blockDim.x / tc;
  const uint4 mu = __ldg(reinterpret_cast<const uint4*>(mean) + cg);
  const uint4 is = __ldg(reinterpret_cast<const uint4*>(invstd) + cg);
  const uint4 ga = __ldg(reinterpret_cast<const uint4*>(gamma) + cg);
  const uint4 be = __ldg(reinterpret_cast<const uint4*>(beta) + cg);
  // two staged rows at a time, four cells of each: eight loads in flight before any use
#pragma unroll 1
  for (int rho0 = 0; rho0 < 2 * kBpT + 1; rho0 += 2) {
    bool rv[2];
    long long rowoff[2];
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const int h = 2 * p0 - 1 + rho0 + e;
      rv[e] = rho0 + e < 2 * kBpT + 1 && h >= 0 && h < H;
      rowoff[e] = ((long long)n * H + (rv[e] ? h : 0)) * W * tc + cg;
    }
    for (int w0 = c0; w0 < W; w0 += 4 * cstep) {
      uint4 xv[2][4];
#pragma unroll
      for (int e = 0; e < 2; ++e)
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int w = w0 + k * cstep;
          xv[e][k] = (rv[e] && w < W) ? __ldg(reinterpret_cast<const uint4*>(x) + rowoff[e] + (long long)w * tc)
                                      : zero4();
        }
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        if (!rv[e]) continue;
        const int rho = rho0 + e;
        uint4* zrow = zs + (rho * W) * tc + cg;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int w = w0 + k * cstep;
          if (w >= W) break;
          const uint4 xh = mul4v(sub4(xv[e][k], mu), is);  // Eq. 1
          uint32_t bits;
          const uint4 z = relu_bits(mul4(add4(mul4v(ga, xh), be), ps), bits);  // Eq. 2, ReLU
          zrow[w * tc] = z;
          if (rho >= 1 && mask) mask[rowoff[e] + (long long)w * tc] = (uint8_t)bits;  // rows 2 p0 .. are this CTA's
        }
      }
    }
  }
  __syncthreads();
#pragma unroll 1
  for (int t = 0; t < kBpT; ++t) {
    const int p = p0 + t;
    if (p >= P) break;
    for (int q = c0; q < Q; q += cstep) {
      // the window's first valid cell (row 2p - 1 and column 2q - 1 are padding at p = 0, q = 0)
      const int r0 = p == 0 ? 1 : 0, s0 = q == 0 ? 1 : 0;
      uint4 m = zs[((2 * t + r0) * W + 2 * q + s0 - 1) * tc + cg];
      uint32_t code[2];
      code[0] = code[1] = (uint32_t)(r0 * 3 + s0) * 0x01010101u;
#pragma unroll
      for (int r = 0; r < 3; ++r) {
        if (2 * p + r - 1 >= H || r < r0) continue;
#pragma unroll
        for (int s2 = 0; s2 < 3; ++s2) {
          const int w = 2 * q + s2 - 1;
          if (w < 0 || w >= W || (r == r0 && s2 <= s0)) continue;
          pool_take(m, code, zs[((2 * t + r) * W + w) * tc + cg], (uint32_t)(r * 3 + s2));
        }
      }
      const long long o = (((long long)n * P + p) * Q + q) * tc + cg;
      reinterpret_cast<uint4*>(pooled)[o] = m;
      reinterpret_cast<uint2*>(codes)[o] = make_uint2(code[0], code[1]);
    }
  }
}

int bn_pool_smem_bytes(int W, int C) { return (2 * kBpT + 1) * W * (C / 8) * 16; }

cudaError_t launch_bn_relu_pool_fwd(const BnLaunch& b, const uint8_t* conv_stats, const uint16_t* x,
                                    const uint16_t* gamma, const uint16_t* beta, uint16_t* mean,
                                    uint16_t* invstd, uint16_t* pooled, uint8_t* codes, uint8_t* mask,
                                    uint16_t* ws, int N, int H, int W, cudaStream_t s) {
  // the statistics as pf16_bn_fwd_bwd's phase 0 takes them (from the conv's
  // partial statistics, or a pass over x), then the fused apply and pooling
  cudaError_t e = conv_stats ? launch_bn_fwd_given_stats(b, conv_stats, x, gamma, beta, nullptr, nullptr, nullptr,
                                                         mean, invstd, s)
                             : launch_bn_fwd(b, x, gamma, beta, nullptr, nullptr, nullptr, mean, invstd, ws, s);
  if (e != cudaSuccess) return e;
  const int C = b.C;
  const int P = (H - 1) / 2 + 1, Q = (W - 1) / 2 + 1;
  const int smem = bn_pool_smem_bytes(W, C);
  // (opted in once for the largest staging the API accepts, 200 KB, whatever this call's size)
  static bool attr[64] = {false};
  if (smem > 200 * 1024) return cudaErrorInvalidValue;
  e = stat_smem_attr(k_bn_relu_pool_fwd, 200 * 1024, attr);
  if (e != cudaSuccess) return e;
  const long long grid = (long long)N * ((P + kBpT - 1) / kBpT);
  const int threads = 256 - 256 % (C / 8);  // a multiple of the channel groups
  launch_pdl(k_bn_relu_pool_fwd, dim3((unsigned)grid), dim3(threads), smem, s, x, gamma, beta,
             static_cast<const uint16_t*>(mean), static_cast<const uint16_t*>(invstd), b.post_scale, pooled, codes,
             mask, N, H, W, C, P, Q);
  return counted_launches(1);
}

// ============================================================================
// Global average pooling (halving tree over hw padded to 2^L, x rn(2^L/hw)).
// ============================================================================
__global__ void k_avgpool_fwd(const uint16_t* __restrict__ x, uint16_t* __restrict__ y, int N, int HW,
                              int C, int levels, uint16_t ratio) {
  pdl_wait();
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
  pdl_wait();
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
  launch_pdl(k_avgpool_fwd, dim3(grid_for(total, 128, 152 * 16)), dim3(128), 0, s, x, y, N, HW, C, L, ratio);
  return counted_launches(1);
}

cudaError_t launch_avgpool_bwd(const uint16_t* dy, uint16_t* dx, int N, int HW, int C,
                               cudaStream_t s) {
  const uint16_t inv = f16_bits_host((float)(1.0 / HW));
  const long long total = (long long)N * HW * (C / 8);
  launch_pdl(k_avgpool_bwd, dim3(grid_for(total, 256, 152 * 16)), dim3(256), 0, s, dy, dx, N, HW, C, inv);
  return counted_launches(1);
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
  pdl_wait();
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
  pdl_wait();
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
  launch_pdl(k_softmax_rows, dim3(B), dim3(kSmThreads), 0, s, logits, bias, labels, K, invB, dlogits, ws);
  launch_pdl(k_softmax_cols, dim3((K + 255) / 256), dim3(256), 0, s, dlogits, ws, B, K, L, ratio, dbias, loss);
  return counted_launches(2);
}

// ============================================================================
// Bounded wait on a device flag: one thread polls *flag (acquire, system
// scope, so a host write through mapped pinned memory is seen as well) until
// it holds `value`, or until limit_ns of %globaltimer time have passed; then it
// records PF16_ERR_TIMEOUT in the status word (the first error stays) and
// returns, so the stream moves on and the context stays usable.
// ============================================================================
__global__ void k_wait_flag(const uint32_t* flag, uint32_t value, unsigned long long limit_ns, int* status) {
  const uint64_t t0 = globaltimer_ns();
  while (true) {
    uint32_t v;
    asm volatile("ld.acquire.sys.global.u32 %0, [%1];" : "=r"(v) : "l"(flag) : "memory");
    if (v == value) return;
    if (globaltimer_ns() - t0 > limit_ns) {
      atomicCAS(status, 0, -7);  // PF16_ERR_TIMEOUT
      return;
    }
    __nanosleep(256);
  }
}

cudaError_t launch_wait_flag(const uint32_t* flag, uint32_t value, unsigned long long limit_ns, int* status,
                             cudaStream_t s) {
  k_wait_flag<<<1, 1, 0, s>>>(flag, value, limit_ns, status);
  return counted_launches(1);
}

}  // namespace pf16
