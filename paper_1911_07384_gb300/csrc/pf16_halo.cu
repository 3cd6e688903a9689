// Wide halo engine: the forward of 3x3 / stride 1 / pad 1 convolutions with
// 128 or 256 output channels over any multiple of 64 input channels, as one
// tcgen05 implicit GEMM whose A operand never goes through TMA im2col.
//
// GEMM rows are the pixels of a padded grid: each padded row holds `ipr`
// images side by side (1, or 4 when the image is narrow), `wi` columns per
// image (at least W + 2), ws = ipr * wi columns in all; a 128-row tile is
// 128 / ws whole padded rows.  For each 64-channel chunk of the input one
// tiled 4-D TMA box brings every input pixel the tile's nine taps read --
// rows i0 - 1 .. i0 + 128/ws, columns -1 .. wi - 2 of each image, zeros
// outside the image -- one pixel per 128-byte swizzled row, so tap (dr, ds)
// is the 128-row window dr * ws + ds pixels into the box (a descriptor start
// moved by whole rows; the 128-byte swizzle is a function of the absolute
// shared address).  The input is read once per tile and chunk instead of
// once per tap, and every load is a plain tiled box: a TMA im2col box of 128
// pixels costs the SM ~700 cycles whatever the MMA work it feeds, which
// bounded the im2col GEMM of these layers.  The weights stream per (chunk,
// tap) through a ring of BN x 64 stages; the accumulators are FP16 in tensor
// memory (kind::f16), two of them, so that a tile's epilogue overlaps the
// next tile's MMAs.  Columns j >= W of the padded grid are computed and then
// dropped by the clipped 4-D TMA store of the output.
//
// Roles as in k_gemm (pf16_gemm.cu): warp 0 the TMA producer, warp 1 the
// TMEM owner and MMA issuer, warps 2-9 the epilogue in two groups, with the
// fused BatchNorm forward statistics of the output optional.  Every mbarrier
// wait is bounded; on expiry the CTA records PF16_ERR_TIMEOUT and all roles
// leave their loops.
#include "pf16_internal.h"
#include "pf16_ptx.cuh"
#include "pf16_epi.cuh"

namespace pf16 {

template <int BN>
struct WideCfg {
  static constexpr int A_SLOT = 32768;  // one input box: at most 256 pixels of 128 bytes
  static constexpr int A_SLOTS = 2;
  static constexpr int B_STAGE = BN * kBK * 2;
  static constexpr int STAGES = BN == 128 ? 8 : 4;
  static constexpr int TMEM_COLS = 2 * BN;
  static constexpr int STAGING_BYTES = kEpiWarps * 4096;
  static constexpr int BAR_BYTES = 8 * (2 * A_SLOTS + 2 * STAGES + 4) + 16;
  // the A slots come first: a tap window's read past its box (at most two
  // rows, feeding only padding columns) stays inside the allocation
  static constexpr int SMEM = 1024 + A_SLOTS * A_SLOT + STAGES * B_STAGE + STAGING_BYTES + BAR_BYTES;
  static_assert(SMEM <= 232448, "shared memory per CTA");
};

// Geometry of tile u: the box origin (coordinates 2 and 3 of the input map)
// and, for a warp's 32 rows, the output image / row / first column.
struct WideTile {
  int img0;  // first image of the tile
  int i0;    // first output row
};

__device__ __forceinline__ WideTile wide_tile(const GemmParams& p, int u) {
  const int rpt = kBM / p.halo_ws;          // padded rows per tile
  const int tpi = p.halo_h / rpt;           // tiles per image (group)
  WideTile t;
  const int g = u / tpi;
  t.i0 = (u - g * tpi) * rpt;
  t.img0 = g * p.halo_ipr;
  return t;
}

// Output pixels of warp `sub`'s 32 rows in tile t: padded row pr, images
// img .. (two images of 16 columns when ipr = 4, else one), first column col0.
struct WideRows {
  int img, i, col0;
  uint32_t vmask;  // rows that are real pixels (column < W)
  int nv;
};

__device__ __forceinline__ WideRows wide_rows(const GemmParams& p, const WideTile& t, int sub) {
  WideRows w;
  const int m = 32 * sub;
  const int pr = m / p.halo_ws, q = m - pr * p.halo_ws;
  w.i = t.i0 + pr;
  if (p.halo_ipr == 1) {
    w.img = t.img0;
    w.col0 = q;
    const int nv = min(32, max(0, p.halo_w - q));
    w.vmask = nv >= 32 ? 0xFFFFFFFFu : (1u << nv) - 1u;
  } else {  // wi = 16: two images per warp
    w.img = t.img0 + q / p.halo_wi;
    w.col0 = 0;
    const uint32_t half = (1u << p.halo_w) - 1u;
    w.vmask = half | (half << 16);
  }
  w.nv = __popc(w.vmask);
  return w;
}

template <int BN>
__global__ void __launch_bounds__(kGemmThreads, 1)
    k_gemm_halo_wide(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB,
                     const __grid_constant__ CUtensorMap mapC, const __grid_constant__ GemmParams p) {
  using Cfg = WideCfg<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* aslots = smem;
  uint8_t* bstages = aslots + Cfg::A_SLOTS * Cfg::A_SLOT;
  uint8_t* staging = bstages + Cfg::STAGES * Cfg::B_STAGE;
  uint64_t* bars = reinterpret_cast<uint64_t*>(staging + Cfg::STAGING_BYTES);
  uint64_t* afull = bars;
  uint64_t* aempty = afull + Cfg::A_SLOTS;
  uint64_t* bfull = aempty + Cfg::A_SLOTS;
  uint64_t* bempty = bfull + Cfg::STAGES;
  uint64_t* tfull = bempty + Cfg::STAGES;
  uint64_t* tempty = tfull + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int ws = p.halo_ws;
  const int chunks = p.halo_chunks;
  const uint32_t box_bytes = (uint32_t)(p.halo_box_rows * ws * 128);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < Cfg::A_SLOTS; ++s) {
      mbar_init(smem_u32(&afull[s]), 1);
      mbar_init(smem_u32(&aempty[s]), 1);
    }
    for (int s = 0; s < Cfg::STAGES; ++s) {
      mbar_init(smem_u32(&bfull[s]), 1);
      mbar_init(smem_u32(&bempty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&tfull[a]), 1);
      mbar_init(smem_u32(&tempty[a]), 4);
    }
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&mapA);
    tma_prefetch_desc(&mapB);
    tma_prefetch_desc(&mapC);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), Cfg::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // set-up done: wait for the kernel this one depends on
  pdl_wait();
  const uint32_t tmem_base = *tmem_slot;
  const int total = p.m_tiles;
  const uint64_t lim = p.wait_limit_ns;

  if (warp == 0) {
    if (lane == 0) {
      int as = 0, bs = 0;
      uint32_t aph = 0, bph = 0, a_issued = 0, b_issued = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < total && !*abort_flag; u += gridDim.x) {
        const WideTile t = wide_tile(p, u);
        // box origin: map coordinates (c, w, h, n) for one image per padded
        // row, (c, w, n, h) for several
        const int c2 = p.halo_ipr == 1 ? t.i0 - 1 : t.img0;
        const int c3 = p.halo_ipr == 1 ? t.img0 : t.i0 - 1;
        for (int cc = 0; ok && cc < chunks; ++cc) {
          if (!mbar_wait(smem_u32(&aempty[as]), aph ^ 1, lim)) {
            ok = false;
            break;
          }
          const uint32_t fa = smem_u32(&afull[as]);
          mbar_arrive_expect_tx(fa, box_bytes);
          tma_load_4d(smem_u32(aslots + as * Cfg::A_SLOT), &mapA, fa, cc * 64, -1, c2, c3);
          ++a_issued;
          if (++as == Cfg::A_SLOTS) {
            as = 0;
            aph ^= 1;
          }
          for (int tp = 0; tp < 9; ++tp) {
            if (!mbar_wait(smem_u32(&bempty[bs]), bph ^ 1, lim)) {
              ok = false;
              break;
            }
            const uint32_t fb = smem_u32(&bfull[bs]);
            const uint32_t dst = smem_u32(bstages + bs * Cfg::B_STAGE);
            mbar_arrive_expect_tx(fb, Cfg::B_STAGE);
            // weights [Cout][9 * Cin]: the tap's 64 input channels of chunk cc
            tma_load_2d(dst, &mapB, fb, p.tap_w[tp] * chunks * 64 + cc * 64, 0);
            ++b_issued;
            if (++bs == Cfg::STAGES) {
              bs = 0;
              bph ^= 1;
            }
          }
        }
      }
      if (!ok) record_timeout(p, abort_flag);
      if (*abort_flag) {
        // let the copies this thread started land before shared memory is released
        uint32_t n = a_issued < (uint32_t)Cfg::A_SLOTS ? a_issued : (uint32_t)Cfg::A_SLOTS;
        int s = as;
        uint32_t ph = aph;
        for (uint32_t i = 0; i < n; ++i) {
          if (--s < 0) {
            s = Cfg::A_SLOTS - 1;
            ph ^= 1;
          }
          mbar_wait(smem_u32(&afull[s]), ph, 1000000000ull);
        }
        n = b_issued < (uint32_t)Cfg::STAGES ? b_issued : (uint32_t)Cfg::STAGES;
        s = bs;
        ph = bph;
        for (uint32_t i = 0; i < n; ++i) {
          if (--s < 0) {
            s = Cfg::STAGES - 1;
            ph ^= 1;
          }
          mbar_wait(smem_u32(&bfull[s]), ph, 1000000000ull);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      int as = 0, bs = 0, acc = 0;
      uint32_t aph = 0, bph = 0, acc_phase = 0;
      // tap windows in 16-byte units, and the two base descriptors
      uint32_t toff[9];
#pragma unroll
      for (int t = 0; t < 9; ++t) toff[t] = (uint32_t)((p.tap_dr[t] * ws + p.tap_ds[t]) * 128) >> 4;
      const uint64_t adesc0 = smem_desc(0, 16, 1024, 2);
      const uint64_t bdesc0 = smem_desc(0, p.b_lbo, p.b_sbo, 2);
      const uint32_t bk16 = (uint32_t)p.b_kstep >> 4;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < total && !*abort_flag; u += gridDim.x) {
        if (!mbar_wait(smem_u32(&tempty[acc]), acc_phase ^ 1, lim)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
        for (int cc = 0; ok && cc < chunks; ++cc) {
          if (!mbar_wait(smem_u32(&afull[as]), aph, lim)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t abase = adesc0 + desc_addr16(smem_u32(aslots + as * Cfg::A_SLOT));
          for (int tp = 0; tp < 9; ++tp) {
            if (!mbar_wait(smem_u32(&bfull[bs]), bph, lim)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint64_t bbase = bdesc0 + desc_addr16(smem_u32(bstages + bs * Cfg::B_STAGE));
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              tc_mma_f16(d_tmem, abase + toff[tp] + kk * 2, bbase + kk * bk16, p.idesc,
                         (cc > 0 || tp > 0 || kk > 0) ? 1u : 0u);
            tc_commit(smem_u32(&bempty[bs]));
            if (++bs == Cfg::STAGES) {
              bs = 0;
              bph ^= 1;
            }
          }
          if (!ok) break;
          tc_commit(smem_u32(&aempty[as]));
          if (++as == Cfg::A_SLOTS) {
            as = 0;
            aph ^= 1;
          }
        }
        if (!ok) break;
        tc_commit(smem_u32(&tfull[acc]));
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1;
      }
      if (!ok) record_timeout(p, abort_flag);
    }
  } else {
    // epilogue warps 2..9: group (w - 2) / 4 drains accumulator 0 or 1 (the
    // CTA's even or odd tiles), warp w its TMEM sub-partition w % 4
    const int e = warp - 2, grp = e >> 2, sub = warp & 3;
    const int acc = grp;
    uint32_t acc_phase = 0;
    const uint32_t stg = smem_u32(staging) + (uint32_t)(e * 4096);
    const bool stats = p.st_mean != nullptr;
    EpiStats st;
    st.init();
    for (int u = blockIdx.x + grp * gridDim.x; u < total; u += 2 * gridDim.x) {
      if (__any_sync(0xffffffffu, *abort_flag != 0)) break;
      const WideTile t = wide_tile(p, u);
      const WideRows w = wide_rows(p, t, sub);
      const bool got = mbar_wait(smem_u32(&tfull[acc]), acc_phase, lim);
      if (!__all_sync(0xffffffffu, got)) {
        if (lane == 0) record_timeout(p, abort_flag);
        break;
      }
      tc_fence_after();
      const uint32_t tbase = tmem_base + ((uint32_t)(sub * 32) << 16) + (uint32_t)(acc * BN);
#pragma unroll 1
      for (int c = 0; c < BN; c += 64) {
        uint32_t r[64];
        tmem_ld16(tbase + c, r);
        tmem_ld16(tbase + c + 16, r + 16);
        tmem_ld16(tbase + c + 32, r + 32);
        tmem_ld16(tbase + c + 48, r + 48);
        tmem_ld_wait();
        if (p.d_f32) f32_to_f16_lo<64>(r);  // FP32 accumulator: one rounding to FP16
        if (c + 64 >= BN) {  // accumulator fully read: hand TMEM back before the stores
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&tempty[acc]));
        }
        if (lane == 0) bulk_wait_read0();  // the previous store has read the staging tile
        __syncwarp();
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          uint4 v;
          v.x = pack_lo(r[j * 8 + 0], r[j * 8 + 1]);
          v.y = pack_lo(r[j * 8 + 2], r[j * 8 + 3]);
          v.z = pack_lo(r[j * 8 + 4], r[j * 8 + 5]);
          v.w = pack_lo(r[j * 8 + 6], r[j * 8 + 7]);
          st_shared_v4(stg + lane * 128 + ((j ^ (lane & 7)) << 4), v);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0 && w.nv > 0) {  // (a box wholly right of the image has nothing to store)
          // output map (c, w, h, n) with 32 x 1 boxes, or (c, w, n, h) with 16 x 2
          if (p.halo_ipr == 1)
            tma_store_4d(&mapC, stg, c, w.col0, w.i, w.img);
          else
            tma_store_4d(&mapC, stg, c, 0, w.img, w.i);
          bulk_commit();
        }
        if (stats && w.nv > 0) st.leafm(c / 64, stg, lane, w.vmask);
      }
      if (stats && w.nv > 0) st.end_tile(w.nv);
      acc_phase ^= 1;
    }
    if (lane == 0) bulk_wait0();
    if (stats) {
      st.write_cta(p, staging, e, blockIdx.x, 0, BN / 64, lane, true);
      if (blockIdx.x == 0 && e == 0 && lane == 0) p.st_hdr[0] = (int)gridDim.x;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, Cfg::TMEM_COLS);
  }
}

template <int BN>
static cudaError_t launch_wide(const CUtensorMap& mA, const CUtensorMap& mB, const CUtensorMap& mC,
                               const GemmParams& p, int grid, cudaStream_t s) {
  static bool attr_set[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 64 && !attr_set[dev]) {
    cudaError_t e = cudaFuncSetAttribute(k_gemm_halo_wide<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         WideCfg<BN>::SMEM);
    if (e != cudaSuccess) return e;
    attr_set[dev] = true;
  }
  launch_pdl(k_gemm_halo_wide<BN>, dim3(grid), dim3(kGemmThreads), WideCfg<BN>::SMEM, s, mA, mB, mC, p);
  return counted_launches(1);
}

cudaError_t launch_gemm_halo_wide(int BN, const CUtensorMap& mA, const CUtensorMap& mB, const CUtensorMap& mC,
                                  const GemmParams& p, int grid, cudaStream_t s) {
  // the input box of a tile must fit its slot, the tile whole padded rows,
  // the tiles whole row groups of an image, and a warp's 32 rows one padded
  // row (one image) or two images of 16 columns
  const int ws = p.halo_ws;
  if (ws <= 0 || kBM % ws != 0 || ws % 32 != 0 || p.halo_ipr * p.halo_wi != ws ||
      (p.halo_ipr != 1 && (p.halo_ipr != 4 || p.halo_wi != 16)) || p.halo_w + 2 > p.halo_wi ||
      p.halo_box_rows != kBM / ws + 2 || p.halo_box_rows * ws * 128 > WideCfg<128>::A_SLOT ||
      p.halo_h % (kBM / ws) != 0 || p.halo_chunks < 1 || p.ntaps != 9 || p.N != BN || p.b_mode != LD_TILED_K)
    return cudaErrorInvalidValue;
  for (int t = 0; t < 9; ++t)
    if (p.tap_dr[t] < 0 || p.tap_dr[t] > 2 || p.tap_ds[t] < 0 || p.tap_ds[t] > 2) return cudaErrorInvalidValue;
  if (p.bs_x) return cudaErrorInvalidValue;  // no backward-statistics epilogue here
  switch (BN) {
    case 128: return launch_wide<128>(mA, mB, mC, p, grid, s);
    case 256: return launch_wide<256>(mA, mB, mC, p, grid, s);
    default: return cudaErrorInvalidValue;
  }
}


// ---------------------------------------------------------------------------
// Weight gradient of the 3x3 / stride 1 / pad 1 convolutions with a multiple
// of 128 output channels K and of 64 input channels C:
//   dW[k][r][s][c] = sum over (n, i, j) of dy[n][i][j][k] * x[n][i+r-1][j+s-1][c].
// The reduction runs over pixels.  A tile is one image row of `nb` images
// side by side, each wi = W + 1 columns wide: a 4-D TMA box (c, w, n, h) of
// wi x nb pixels (at most 128), one 128-byte swizzled row per pixel.  The dy
// box starts at column 0 (column W reads as zero); the input box starts at
// column -1 and row h + r - 1, so box pixel q holds x at column (q mod wi) - 1
// and the window one to two pixels further holds the taps s = 1, 2 of the
// same dy pixel.  A window that runs past an image's columns meets the next
// image's column -1 (zero) or a dy column >= W (zero); past the last image it
// reads a zero tail of shared memory that no copy ever writes (dy rows and
// input pixels past the box are zeroed once at start).  One MMA (M = 128
// output channels, N = 192, K = 16 pixels, both operands MN-major):
//   A = dy, two 64-channel atoms (the two dy boxes, 16 KB apart);
//   B = the input at three windows one pixel apart (s = 0, 1, 2; LBO 128 B,
//       a descriptor start moved by whole 128-byte rows).
// A unit is (chunk of tiles, output-channel tile kt, input chunk cc, filter
// row r): its 128 x 192 FP16 accumulator (kind::f16 in tensor memory, two of
// them so that a unit's drain overlaps the next unit's MMAs) sums the chunk's
// pixels, and the epilogue writes it as rows k, columns (r*3 + s)*C + cc*64 +
// c of the chunk's partial plane [K][9*C] -- the weight gradient's own
// layout, so the split-K tree (k_splitk_reduce) writes dw directly.  Units
// run chunk-major, so the SMs at work at one time read the same few chunks
// of dy and x from L2.  The input is read 3 x K/128 times and dy 3 x C/64
// times, all from L2, against 9 x K/128 input reads through TMA im2col boxes
// in the im2col GEMM.  Non-finite inputs: a dy of zero at a padding column
// meets a real input pixel (column 0 of the next image), so an infinite or
// NaN input there gives NaN in the s = 2 taps.
// Roles: warp 0 the TMA producer, warp 1 the TMEM owner and MMA issuer,
// warps 2-5 the epilogue (TMEM sub-partition warp % 4).  Every mbarrier wait
// is bounded; on expiry the CTA records PF16_ERR_TIMEOUT and all roles leave.
// ---------------------------------------------------------------------------
struct WideWgradCfg {
  static constexpr int DY_BYTES = 2 * 16384;  // 128 pixels x 128 output channels: two 64-channel boxes
  static constexpr int X_BYTES = 16384 + 1024;  // 128 input pixels, then the zero tail windows read into
  static constexpr int STAGE = DY_BYTES + X_BYTES;
  static constexpr int STAGES = 4;
  static constexpr int ACC_COLS = 192;
  static constexpr int TMEM_COLS = 512;  // accumulators at columns 0 and 192
  static constexpr int BAR_BYTES = 8 * (2 * STAGES + 4) + 16;
  static constexpr int SMEM = 1024 + STAGES * STAGE + BAR_BYTES;
  static_assert(STAGE % 1024 == 0, "stage bases keep the 1024-byte alignment of the 128-byte swizzle");
  static_assert(SMEM <= 232448, "shared memory per CTA");
};
constexpr int kWideWgradThreads = 192;

// Unit u: chunk q = u / types, then filter row r, input chunk cc and
// output-channel tile kt (r fastest).
struct WideWgradUnit {
  int q, r, cc, kt, t0, t1;
};

__device__ __forceinline__ WideWgradUnit wide_wgrad_unit(const GemmParams& p, int u) {
  const int types = 3 * p.halo_chunks * (p.M / 128);
  WideWgradUnit w;
  w.q = u / types;
  int ty = u - w.q * types;
  w.r = ty % 3;
  ty /= 3;
  w.cc = ty % p.halo_chunks;
  w.kt = ty / p.halo_chunks;
  w.t0 = w.q * p.kb_per_split;
  w.t1 = min(p.num_kb, w.t0 + p.kb_per_split);
  return w;
}

__global__ void __launch_bounds__(kWideWgradThreads, 1)
    k_wgrad3x3_wide(const __grid_constant__ CUtensorMap mapDy, const __grid_constant__ CUtensorMap mapX,
                    const __grid_constant__ GemmParams p) {
  using Cfg = WideWgradCfg;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Cfg::STAGES * Cfg::STAGE);
  uint64_t* full = bars;
  uint64_t* empty = full + Cfg::STAGES;
  uint64_t* tfull = empty + Cfg::STAGES;
  uint64_t* tempty = tfull + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // zero the stages once: rows past a box are never written by a copy
  for (int i = threadIdx.x; i < Cfg::STAGES * Cfg::STAGE / 16; i += blockDim.x)
    st_shared_v4(smem_u32(smem) + (uint32_t)(i * 16), make_uint4(0u, 0u, 0u, 0u));
  fence_proxy_async_smem();
  if (threadIdx.x == 0) {
    for (int s = 0; s < Cfg::STAGES; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&tfull[a]), 1);
      mbar_init(smem_u32(&tempty[a]), 4);
    }
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&mapDy);
    tma_prefetch_desc(&mapX);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), Cfg::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_wait();
  const uint32_t tmem_base = *tmem_slot;
  const int total = p.m_tiles;  // units
  const int H = p.halo_h, nb = p.halo_ipr;
  const uint32_t box_bytes = (uint32_t)(p.halo_wi * nb * 128);
  const uint64_t lim = p.wait_limit_ns;

  if (warp == 0) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0, issued = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < total && !*abort_flag; u += gridDim.x) {
        const WideWgradUnit w = wide_wgrad_unit(p, u);
        for (int t = w.t0; t < w.t1; ++t) {
          const int g = t / H, h = t - g * H;
          if (!mbar_wait(smem_u32(&empty[stage]), phase ^ 1, lim)) {
            ok = false;
            break;
          }
          const uint32_t fb = smem_u32(&full[stage]);
          const uint32_t dst = smem_u32(smem + stage * Cfg::STAGE);
          mbar_arrive_expect_tx(fb, 3 * box_bytes);
          // maps (c, w, n, h): dy from column 0 of row h, the input from
          // column -1 of row h + r - 1 (rows and columns outside read zero)
          tma_load_4d(dst, &mapDy, fb, w.kt * 128, 0, g * nb, h);
          tma_load_4d(dst + 16384, &mapDy, fb, w.kt * 128 + 64, 0, g * nb, h);
          tma_load_4d(dst + Cfg::DY_BYTES, &mapX, fb, w.cc * 64, -1, g * nb, h + w.r - 1);
          ++issued;
          if (++stage == Cfg::STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (!ok) record_timeout(p, abort_flag);
      if (*abort_flag) {  // let every copy this thread started land before the CTA can exit
        const uint32_t nn = issued < (uint32_t)Cfg::STAGES ? issued : (uint32_t)Cfg::STAGES;
        int s = stage;
        uint32_t ph = phase;
        for (uint32_t i = 0; i < nn; ++i) {
          if (--s < 0) {
            s = Cfg::STAGES - 1;
            ph ^= 1;
          }
          mbar_wait(smem_u32(&full[s]), ph, 1000000000ull);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // A: dy, MN-major, two 64-channel atoms 16 KB apart, 8-pixel K groups
      // 1 KB apart; B: the input, three 64-channel atoms one pixel apart
      const uint64_t adesc0 = smem_desc(0, 16384, 1024, 2);
      const uint64_t bdesc0 = smem_desc(0, 128, 1024, 2);
      int stage = 0, acc = 0;
      uint32_t phase = 0, acc_phase = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < total && !*abort_flag; u += gridDim.x) {
        const WideWgradUnit w = wide_wgrad_unit(p, u);
        if (!mbar_wait(smem_u32(&tempty[acc]), acc_phase ^ 1, lim)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * Cfg::ACC_COLS);
        for (int t = w.t0; t < w.t1; ++t) {
          if (!mbar_wait(smem_u32(&full[stage]), phase, lim)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa16 = desc_addr16(smem_u32(smem + stage * Cfg::STAGE));
          const uint64_t ab = adesc0 + sa16;
          const uint64_t bb = bdesc0 + sa16 + (uint32_t)(Cfg::DY_BYTES >> 4);
#pragma unroll
          for (int js = 0; js < 8; ++js)  // 16 pixels (2 KB of each operand) per MMA
            tc_mma_f16(d_tmem, ab + (uint32_t)(js * 128), bb + (uint32_t)(js * 128), p.idesc,
                       (t > w.t0 || js > 0) ? 1u : 0u);
          tc_commit(smem_u32(&empty[stage]));
          if (++stage == Cfg::STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        tc_commit(smem_u32(&tfull[acc]));
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1;
      }
      if (!ok) record_timeout(p, abort_flag);
    }
  } else {
    // epilogue warps 2..5: TMEM sub-partition warp % 4 holds output channels
    // kt * 128 + 32 * (warp % 4) + lane; a lane writes its channel's three
    // 64-wide runs (s = 0, 1, 2) of the unit's filter row
    const int sub = warp & 3;
    const int C = p.halo_chunks * 64;
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int u = blockIdx.x; u < total; u += gridDim.x) {
      if (__any_sync(0xffffffffu, *abort_flag != 0)) break;
      const WideWgradUnit w = wide_wgrad_unit(p, u);
      const bool got = mbar_wait(smem_u32(&tfull[acc]), acc_phase, lim);
      if (!__all_sync(0xffffffffu, got)) {
        if (lane == 0) record_timeout(p, abort_flag);
        break;
      }
      tc_fence_after();
      const int k = w.kt * 128 + sub * 32 + lane;
      uint16_t* prow = p.out + ((size_t)w.q * p.M + k) * (size_t)p.ldo + (size_t)(w.r * 3) * C + w.cc * 64;
#pragma unroll 1
      for (int s = 0; s < 3; ++s) {
        const uint32_t tb =
            tmem_base + ((uint32_t)(sub * 32) << 16) + (uint32_t)(acc * Cfg::ACC_COLS + s * 64);
        uint32_t v[64];
        tmem_ld16(tb, v);
        tmem_ld16(tb + 16, v + 16);
        tmem_ld16(tb + 32, v + 32);
        tmem_ld16(tb + 48, v + 48);
        tmem_ld_wait();
        if (p.d_f32) f32_to_f16_lo<64>(v);  // FP32 accumulator: one rounding to FP16
        if (s == 2) {  // accumulator fully read: hand it back before the stores
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&tempty[acc]));
        }
        uint4* dst = reinterpret_cast<uint4*>(prow + (size_t)s * C);
#pragma unroll
        for (int j = 0; j < 8; ++j)
          dst[j] = make_uint4(pack_lo(v[j * 8 + 0], v[j * 8 + 1]), pack_lo(v[j * 8 + 2], v[j * 8 + 3]),
                              pack_lo(v[j * 8 + 4], v[j * 8 + 5]), pack_lo(v[j * 8 + 6], v[j * 8 + 7]));
      }
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, Cfg::TMEM_COLS);
  }
}

cudaError_t launch_wgrad3x3_wide(const CUtensorMap& mDy, const CUtensorMap& mX, const GemmParams& p, int grid,
                                 cudaStream_t s) {
  // a box of at most 128 pixels with one zero column between images, whole
  // 128-channel output tiles and 64-channel input chunks, and every unit of
  // the plan non-empty (chunks * per_chunk covers the tiles, the last chunk
  // starting inside them)
  const int types = p.M > 0 && p.M % 128 == 0 ? 3 * p.halo_chunks * (p.M / 128) : 0;
  if (types < 3 || p.halo_chunks < 1 || p.halo_wi < p.halo_w + 1 || p.halo_w < 1 || p.halo_ipr < 1 ||
      p.halo_wi * p.halo_ipr > 128 || p.halo_h < 1 || p.num_kb < 1 || p.kb_per_split < 1 || p.splits < 1 ||
      p.m_tiles != p.splits * types || (long long)(p.splits - 1) * p.kb_per_split >= p.num_kb ||
      (long long)p.splits * p.kb_per_split < p.num_kb || p.ldo != 9LL * p.halo_chunks * 64 || grid < 1)
    return cudaErrorInvalidValue;
  static bool attr_set[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 64 && !attr_set[dev]) {
    cudaError_t e = cudaFuncSetAttribute(k_wgrad3x3_wide, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         WideWgradCfg::SMEM);
    if (e != cudaSuccess) return e;
    attr_set[dev] = true;
  }
  launch_pdl(k_wgrad3x3_wide, dim3(grid), dim3(kWideWgradThreads), WideWgradCfg::SMEM, s, mDy, mX, p);
  return counted_launches(1);
}
}  // namespace pf16
