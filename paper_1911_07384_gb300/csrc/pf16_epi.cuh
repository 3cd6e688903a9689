// Shared pieces of the tcgen05 conv engines (pf16_gemm.cu, pf16_halo.cu):
// the warp-role constants, the bounded-wait abort, and the epilogue's
// packing and fused BatchNorm statistics (forward and backward leaves).
// Device code only; included inside namespace pf16 by each engine.
#pragma once
#include "pf16_internal.h"
#include "pf16_ptx.cuh"

namespace pf16 {

// Epilogue: two warps per TMEM sub-partition (lanes 32*(warp % 4) ...), warps
// 2-5 draining accumulator 0 (the CTA's even tiles) and warps 6-9 accumulator 1
// (its odd tiles), so two tiles drain at once.
constexpr int kEpiWarps = 8;
constexpr int kGemmThreads = 32 * (2 + kEpiWarps);
// The wide epilogue of k_gemm (WE, plain epilogue of short reductions): 16
// warps, two per TMEM sub-partition and accumulator, each draining one column
// half of the tile.
constexpr int kEpiWarpsWide = 16;
constexpr int kGemmThreadsWide = 32 * (2 + kEpiWarpsWide);
// XF (BatchNorm in the operand path): eight transform warps after the epilogue's
constexpr int kXfWarp0 = 2 + kEpiWarps;
constexpr int kXfWarps = 8;
constexpr int kGemmThreadsXf = kGemmThreads + 32 * kXfWarps;

static constexpr int kErrTimeout = -7;  // PF16_ERR_TIMEOUT

__device__ __forceinline__ void record_timeout(const GemmParams& p, volatile int* abort_flag) {
  *abort_flag = 1;
  atomicCAS(p.status, 0, kErrTimeout);
}

// low halves of two 32-bit TMEM words -> one f16x2
__device__ __forceinline__ uint32_t pack_lo(uint32_t a, uint32_t b) { return __byte_perm(a, b, 0x5410); }
// FP32 accumulator words -> binary16 (roundTiesToEven) in their low 16 bits, in place
template <int N>
__device__ __forceinline__ void f32_to_f16_lo(uint32_t* r) {
#pragma unroll
  for (int i = 0; i < N; ++i) r[i] = __half_as_ushort(__float2half_rn(__uint_as_float(r[i])));
}


// ---------------------------------------------------------------------------
// Fused BatchNorm forward statistics of the output (GemmParams::st_mean).
// After a warp has staged its 32 rows x 64 columns, lane l reduces channel
// pair (2l, 2l+1) over the warp's valid rows (a prefix of the 32, or any subset
// given as a row mask): the mean
// of the 32-leaf halving tree (zero padded, scaled by rn(32/n) when rows are
// missing) and, over the same rows, the mean squared deviation from it.  The
// leaf is pushed into the warp's binary-counter stack of (mean, variance,
// count) nodes merged by the count-aware parallel-variance rule -- the
// arithmetic of the BatchNorm statistics kernels -- and the stack is closed
// once, after the warp's last tile.  All binary16, one rounding per op.
// ---------------------------------------------------------------------------
constexpr int kStChunks = 4;   // 64-column chunks of a tile (BN <= 256)
constexpr int kStLevels = kMaxTileTreeLevels;  // tiles per warp below 2^12

__device__ __forceinline__ uint32_t hmerge2f(uint32_t a, uint32_t b) {  // rn(a/2 + rn(b/2))
  return hfma2_rn(a, 0x38003800u, hmul2_rn(b, 0x38003800u));
}
__device__ __forceinline__ uint32_t dup2h(uint16_t h) { return (uint32_t)h | ((uint32_t)h << 16); }

// node a <- merge(a, b) with counts na, nb (the result's count is na + nb)
__device__ __forceinline__ void mv2_merge(uint32_t& amu, uint32_t& av, int na, uint32_t bmu, uint32_t bv,
                                          int nb) {
  if (nb == 0) return;
  if (na == 0) {
    amu = bmu;
    av = bv;
    return;
  }
  const uint32_t d = hsub2_rn(bmu, amu);
  if (na == nb) {
    const uint32_t dh = hmul2_rn(d, 0x38003800u);
    amu = hmerge2f(amu, bmu);
    av = hadd2_rn(hmerge2f(av, bv), hmul2_rn(dh, dh));
  } else {
    const float n = (float)(na + nb);
    const uint32_t wa = dup2h(__half_as_ushort(__float2half_rn(__fdiv_rn((float)na, n))));
    const uint32_t wb = dup2h(__half_as_ushort(__float2half_rn(__fdiv_rn((float)nb, n))));
    const uint32_t wab = hmul2_rn(wa, wb);
    amu = hadd2_rn(hmul2_rn(amu, wa), hmul2_rn(bmu, wb));
    av = hadd2_rn(hadd2_rn(hmul2_rn(av, wa), hmul2_rn(bv, wb)), hmul2_rn(hmul2_rn(d, d), wab));
  }
}

struct EpiStats {
  uint32_t mu[kStChunks][kStLevels], v[kStChunks][kStLevels];
  int n[kStLevels];
  unsigned cnt;

  __device__ __forceinline__ void init() { cnt = 0; }

  // leaf of chunk c from the staged tile (row r at stg + r*128, 128B-swizzled)
  // over the warp's first nv rows
  __device__ __forceinline__ void leaf(int c, uint32_t stg, int lane, int nv) {
    if (nv == 32)  // a full leaf (every tile but a tensor's last): no row tests
      leaf_impl<true, false>(c, stg, lane, 0xFFFFFFFFu, 32);
    else
      leaf_impl<false, false>(c, stg, lane, 0u, nv);
  }
  // the same over the rows whose bit is set in vmask (non-zero); for a prefix
  // mask this is leaf() exactly
  __device__ __forceinline__ void leafm(int c, uint32_t stg, int lane, uint32_t vmask) {
    if (vmask == 0xFFFFFFFFu)
      leaf_impl<true, true>(c, stg, lane, vmask, 32);
    else
      leaf_impl<false, true>(c, stg, lane, vmask, __popc(vmask));
  }
  // MASK: rows tested against vmask bit by bit; else the first nv rows
  template <bool FULL, bool MASK>
  __device__ __forceinline__ void leaf_impl(int c, uint32_t stg, int lane, uint32_t vmask, int nv) {
    const uint32_t col = (uint32_t)(lane & 3) * 4;
    uint32_t x[32], t[32];  // the 32 rows' channel pair, read once
#pragma unroll
    for (int r = 0; r < 32; ++r) {
      asm volatile("ld.shared.b32 %0, [%1];" : "=r"(x[r]) : "r"(stg + r * 128 + ((((uint32_t)lane >> 2) ^ (r & 7)) << 4) + col));
      t[r] = (FULL || (MASK ? ((vmask >> r) & 1u) != 0 : r < nv)) ? x[r] : 0u;
    }
#pragma unroll
    for (int w = 16; w >= 1; w /= 2)
#pragma unroll
      for (int i = 0; i < w; ++i) t[i] = hmerge2f(t[2 * i], t[2 * i + 1]);
    uint32_t mu = t[0], sc = 0;
    if (!FULL && nv < 32) {
      sc = dup2h(__half_as_ushort(__float2half_rn(32.0f / (float)nv)));
      mu = hmul2_rn(mu, sc);
    }
#pragma unroll
    for (int r = 0; r < 32; ++r) {
      const uint32_t e = hsub2_rn(x[r], mu);
      t[r] = (FULL || (MASK ? ((vmask >> r) & 1u) != 0 : r < nv)) ? hmul2_rn(e, e) : 0u;
    }
#pragma unroll
    for (int w = 16; w >= 1; w /= 2)
#pragma unroll
      for (int i = 0; i < w; ++i) t[i] = hmerge2f(t[2 * i], t[2 * i + 1]);
    uint32_t var = t[0];
    if (!FULL && nv < 32) var = hmul2_rn(var, sc);
    // push into chunk c's stack (counts are updated by end_tile)
    int nn = nv;
#pragma unroll 1
    for (int l = 0; l < kStLevels; ++l) {
      if (cnt & (1u << l)) {
        uint32_t m2 = this->mu[c][l], v2 = this->v[c][l];
        mv2_merge(m2, v2, n[l], mu, var, nn);
        mu = m2;
        var = v2;
        nn += n[l];
      } else {
        this->mu[c][l] = mu;
        this->v[c][l] = var;
        break;
      }
    }
  }
  // after all chunks of a tile with nv valid rows
  __device__ __forceinline__ void end_tile(int nv) {
    int nn = nv;
#pragma unroll 1
    for (int l = 0; l < kStLevels; ++l) {
      if (cnt & (1u << l)) {
        nn += n[l];
      } else {
        n[l] = nn;
        break;
      }
    }
    ++cnt;
  }
  // Close the stacks, merge the CTA's 8 epilogue warps (a balanced tree over
  // warps 0..7, in shared memory `sm`, >= 8.3 KB, free of pending TMA reads)
  // and write the CTA's node as `slot` for chunks c < nchunks.  Called by all
  // ew epilogue warps; uses named barrier 1.  With the wide epilogue (ew = 16)
  // warps 8h .. 8h + 7 hold the chunks of column half h (cph chunks each), and
  // chunk c is merged over the eight warps of its half, in the same tree.
  __device__ __forceinline__ void write_cta(const GemmParams& p, uint8_t* sm, int e, int slot, int n0,
                                            int nchunks, int lane, bool write_count, int ew = kEpiWarps,
                                            int cph = kStChunks) {
    uint32_t* node = reinterpret_cast<uint32_t*>(sm);                // [ew][kStChunks][32][2]
    int* ncnt = reinterpret_cast<int*>(sm + ew * kStChunks * 32 * 8);  // [ew]
    asm volatile("bar.sync 1, %0;" ::"r"(32 * ew) : "memory");
    int total = 0;
    for (int c = 0; c < nchunks; ++c) {
      if (ew > 8 && c / cph != (e >> 3)) continue;  // a chunk of the other column half
      uint32_t am = 0, av = 0;
      int an = 0;
#pragma unroll 1
      for (int l = 0; l < kStLevels; ++l) {
        if (cnt & (1u << l)) {
          uint32_t m2 = mu[c][l], v2 = v[c][l];
          mv2_merge(m2, v2, n[l], am, av, an);
          am = m2;
          av = v2;
          an += n[l];
        }
      }
      node[((e * kStChunks + c) * 32 + lane) * 2] = am;
      node[((e * kStChunks + c) * 32 + lane) * 2 + 1] = av;
      total = an;
    }
    if (lane == 0) ncnt[e] = total;
    asm volatile("bar.sync 1, %0;" ::"r"(32 * ew) : "memory");
    if (e != 0) return;
    int tot = 0;
    for (int c = 0; c < nchunks; ++c) {
      uint32_t m[8], vv[8];
      int nn[8];
      const int w0 = ew > 8 ? 8 * (c / cph) : 0;
#pragma unroll
      for (int w = 0; w < 8; ++w) {
        m[w] = node[(((w0 + w) * kStChunks + c) * 32 + lane) * 2];
        vv[w] = node[(((w0 + w) * kStChunks + c) * 32 + lane) * 2 + 1];
        nn[w] = ncnt[w0 + w];
      }
#pragma unroll
      for (int h = 1; h < 8; h *= 2)
#pragma unroll
        for (int w = 0; w < 8; w += 2 * h) {
          mv2_merge(m[w], vv[w], nn[w], m[w + h], vv[w + h], nn[w + h]);
          nn[w] += nn[w + h];
        }
      const long long o = (long long)slot * p.N + n0 + c * 64 + 2 * lane;
      *reinterpret_cast<uint32_t*>(p.st_mean + o) = m[0];
      *reinterpret_cast<uint32_t*>(p.st_var + o) = vv[0];
      tot = nn[0];
    }
    if (write_count && lane == 0) p.st_cnt[slot] = tot;
  }

  // Backward statistics (GemmParams::bs_x): leaf of chunk c from the staged
  // gradient tile g and the prefetched inputs of its 32 rows (BwdIn).  Lane l
  // takes channel pair (2l, 2l+1): dy' = g where the ReLU passed and
  // dy' * rn(rn(x - mean) * invstd); rows r >= nv are zero leaves.  Each
  // 32-leaf pairwise sum is pushed into chunk c's binary counter of sum nodes
  // (mu: dy', v: dy' xhat).
  __device__ __forceinline__ void leaf_bwd(int c, uint32_t stg, int lane, int nv, const struct BwdIn& in);
  // The same leaf with x read from a 128B-swizzled 32 x 64 tile at xs (laid
  // out as the staged tile), ReLU bits m of row `lane` and the pair's mean2 /
  // invstd2.
  __device__ __forceinline__ void leaf_bwd_tile(int c, uint32_t stg, uint32_t xs, int lane, int nv, uint2 m,
                                                uint32_t mean2, uint32_t invstd2);
  template <class XF>
  __device__ __forceinline__ void leaf_bwd_core(int c, uint32_t stg, int lane, int nv, uint2 m, uint32_t mean2,
                                                uint32_t invstd2, XF xf);
  template <bool FULL, class XF>
  __device__ __forceinline__ void leaf_bwd_impl(int c, uint32_t stg, int lane, int nv, uint2 m, uint32_t mean2,
                                                uint32_t invstd2, XF xf);
  // Close the backward counters as if zero leaves padded them to 2^levels,
  // add the CTA's 8 epilogue warps' sums (warps 0..7 in a balanced tree,
  // through `sm` as write_cta) and write the CTA's sums as `slot`.
  __device__ __forceinline__ void write_cta_bwd(const GemmParams& p, uint8_t* sm, int e, int slot, int n0,
                                                int nchunks, int lane, int levels) {
    uint32_t* node = reinterpret_cast<uint32_t*>(sm);  // [8][kStChunks][32][2]
    asm volatile("bar.sync 1, %0;" ::"r"(32 * kEpiWarps) : "memory");
    for (int c = 0; c < nchunks; ++c) {
      uint32_t a1 = 0, a2 = 0;
      bool have = false;
#pragma unroll 1
      for (int l = 0; l <= levels && l < kStLevels; ++l) {
        if (l == levels) {
          if (!have && (cnt & (1u << l))) {  // exactly 2^levels leaves
            a1 = this->mu[c][l];
            a2 = this->v[c][l];
          }
        } else if (cnt & (1u << l)) {
          a1 = hadd2_rn(this->mu[c][l], have ? a1 : 0u);
          a2 = hadd2_rn(this->v[c][l], have ? a2 : 0u);
          have = true;
        } else if (have) {
          a1 = hadd2_rn(a1, 0u);
          a2 = hadd2_rn(a2, 0u);
        }
      }
      node[((e * kStChunks + c) * 32 + lane) * 2] = a1;
      node[((e * kStChunks + c) * 32 + lane) * 2 + 1] = a2;
    }
    asm volatile("bar.sync 1, %0;" ::"r"(32 * kEpiWarps) : "memory");
    if (e != 0) return;
    for (int c = 0; c < nchunks; ++c) {
      uint32_t m1[8], m2[8];
#pragma unroll
      for (int w = 0; w < 8; ++w) {
        m1[w] = node[((w * kStChunks + c) * 32 + lane) * 2];
        m2[w] = node[((w * kStChunks + c) * 32 + lane) * 2 + 1];
      }
#pragma unroll
      for (int h = 1; h < 8; h *= 2)
#pragma unroll
        for (int w = 0; w < 8; w += 2 * h) {
          m1[w] = hadd2_rn(m1[w], m1[w + h]);
          m2[w] = hadd2_rn(m2[w], m2[w + h]);
        }
      const long long o = (long long)slot * p.N + n0 + c * 64 + 2 * lane;
      *reinterpret_cast<uint32_t*>(p.st_mean + o) = m1[0];
      *reinterpret_cast<uint32_t*>(p.st_var + o) = m2[0];
    }
  }
};

// Inputs of one backward leaf, loaded ahead of the tile's accumulator so that
// their latency overlaps the wait for it: for the warp's 32 rows starting at
// row0 of [rows][N] (pixels in order) and the 64 columns at col0, lane l
// holds x of channel pair (2l, 2l+1) for every row, and the 64 ReLU bits of
// row l (all ones without a mask); plus the pair's mean and invstd.
struct BwdIn {
  uint32_t x[32];
  uint2 m;
  uint32_t mu2, is2;

  __device__ __forceinline__ void load(const GemmParams& p, long long row0, int col0, int nv, int lane) {
    const uint16_t* xr = p.bs_x + row0 * p.ldo + col0;
#pragma unroll
    for (int r = 0; r < 32; ++r)
      x[r] = r < nv ? __ldg(reinterpret_cast<const uint32_t*>(xr + r * p.ldo) + lane) : 0u;
    m = make_uint2(0xFFFFFFFFu, 0xFFFFFFFFu);
    if (p.bs_mask && lane < nv)
      m = __ldg(reinterpret_cast<const uint2*>(p.bs_mask + (row0 + lane) * (p.N / 8) + col0 / 8));
    mu2 = __ldg(reinterpret_cast<const uint32_t*>(p.bs_mean + col0) + lane);
    is2 = __ldg(reinterpret_cast<const uint32_t*>(p.bs_invstd + col0) + lane);
  }
};

template <class XF>
__device__ __forceinline__ void EpiStats::leaf_bwd_core(int c, uint32_t stg, int lane, int nv, uint2 m,
                                                        uint32_t mean2, uint32_t invstd2, XF xf) {
  if (nv == 32)  // a full leaf: no row tests
    leaf_bwd_impl<true>(c, stg, lane, nv, m, mean2, invstd2, xf);
  else
    leaf_bwd_impl<false>(c, stg, lane, nv, m, mean2, invstd2, xf);
}

template <bool FULL, class XF>
__device__ __forceinline__ void EpiStats::leaf_bwd_impl(int c, uint32_t stg, int lane, int nv, uint2 m,
                                                        uint32_t mean2, uint32_t invstd2, XF xf) {
  const uint32_t col = (uint32_t)(lane & 3) * 4;
  uint32_t t1[32], t2[32];
#pragma unroll
  for (int r = 0; r < 32; ++r) {
    const uint32_t off = r * 128 + ((((uint32_t)lane >> 2) ^ (r & 7)) << 4) + col;
    uint32_t g;
    asm volatile("ld.shared.b32 %0, [%1];" : "=r"(g) : "r"(stg + off));
    // row r's ReLU bits from lane r; this lane's two channels are bits 2l, 2l+1
    const uint32_t mlo = __shfl_sync(0xffffffffu, m.x, r), mhi = __shfl_sync(0xffffffffu, m.y, r);
    const uint32_t b = (lane < 16 ? mlo >> (2 * lane) : mhi >> (2 * lane - 32)) & 3u;
    const uint32_t mk = ((b & 1u) ? 0x0000FFFFu : 0u) | ((b & 2u) ? 0xFFFF0000u : 0u);
    const uint32_t d = (FULL || r < nv) ? (g & mk) : 0u;
    t1[r] = d;
    t2[r] = (FULL || r < nv) ? hmul2_rn(d, hmul2_rn(hsub2_rn(xf(r, off), mean2), invstd2)) : 0u;
  }
#pragma unroll
  for (int w = 16; w >= 1; w /= 2)
#pragma unroll
    for (int i = 0; i < w; ++i) {
      t1[i] = hadd2_rn(t1[2 * i], t1[2 * i + 1]);
      t2[i] = hadd2_rn(t2[2 * i], t2[2 * i + 1]);
    }
  uint32_t n1 = t1[0], n2 = t2[0];
#pragma unroll 1
  for (int l = 0; l < kStLevels; ++l) {
    if (cnt & (1u << l)) {
      n1 = hadd2_rn(mu[c][l], n1);
      n2 = hadd2_rn(v[c][l], n2);
    } else {
      mu[c][l] = n1;
      v[c][l] = n2;
      break;
    }
  }
}

__device__ __forceinline__ void EpiStats::leaf_bwd(int c, uint32_t stg, int lane, int nv, const BwdIn& in) {
  leaf_bwd_core(c, stg, lane, nv, in.m, in.mu2, in.is2, [&](int r, uint32_t) { return in.x[r]; });
}

__device__ __forceinline__ void EpiStats::leaf_bwd_tile(int c, uint32_t stg, uint32_t xs, int lane, int nv, uint2 m,
                                                        uint32_t mean2, uint32_t invstd2) {
  leaf_bwd_core(c, stg, lane, nv, m, mean2, invstd2, [&](int, uint32_t off) {
    uint32_t x;
    asm volatile("ld.shared.b32 %0, [%1];" : "=r"(x) : "r"(xs + off));
    return x;
  });
}

}  // namespace pf16
