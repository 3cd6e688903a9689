// tcgen05 implicit-GEMM engine for the pure-FP16 convolutions (forward, data
// gradient, weight gradient) of the ResNet-50 training step: FP16 operands,
// FP16 accumulation in tensor memory, FP16 results -- no FP32 anywhere
// (paper Sec. 5.2: all arithmetic and storage in FP16).
//
// One persistent CTA per SM, 10 warps:
//   warp 0    TMA producer: one elected lane streams 64-wide K-blocks of A
//             and B into a ring of shared-memory stages (mbarrier full/empty).
//   warp 1    allocates tensor memory; one lane issues tcgen05.mma
//             (kind::f16, D = f16, M = 128, N = BN, K = 16) and commits each
//             stage back to the producer and each finished tile to the
//             epilogue.  Two TMEM accumulators alternate so the epilogue of
//             tile i overlaps the MMAs of tile i + 1.
//   warps 2-9 epilogue, two groups of four: group g drains accumulator g (the
//             CTA's even or odd tiles), warp w its TMEM sub-partition w % 4;
//             tcgen05.ld of one accumulator row per thread, pack to FP16,
//             stage in shared memory and store by TMA (or FP16-accumulate, or
//             write a split-K partial), with the fused BatchNorm statistics.
// Every mbarrier wait is bounded; on expiry the CTA records PF16_ERR_TIMEOUT
// and all roles leave their loops, so the kernel always terminates.
#include <cstdio>

#include "pf16_internal.h"
#include "pf16_ptx.cuh"
#include "pf16_epi.cuh"

namespace pf16 {


// TMAE: the TMA-fed backward-statistics epilogue keeps four 32 x 64 tiles per
// warp (two staging tiles, two BatchNorm-input tiles, filled by TMA a chunk
// ahead), paid for with pipeline stages; plus two transaction barriers per warp.
// WE: the wide epilogue (16 warps, 4 KB of staging each), paid for with
// pipeline stages -- it serves short reductions, whose few K-blocks per tile
// need few stages.
template <int BN, bool TMAE = false, bool XF = false, bool WE = false>
struct GemmCfg {
  static constexpr int A_BYTES = kBM * kBK * 2;
  static constexpr int B_BYTES = BN * kBK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int STAGES = WE ? (BN == 128 ? 5 : 3)
                                   : TMAE ? (BN == 64 ? 4 : (BN == 128 ? 3 : 2)) : (BN == 64 ? 8 : (BN == 128 ? 6 : 4));
  static constexpr int TMEM_COLS = 2 * BN <= 128 ? 128 : (2 * BN <= 256 ? 256 : 512);
  static constexpr int EW = WE ? kEpiWarpsWide : kEpiWarps;  // epilogue warps
  static constexpr int WARP_BUF = TMAE ? 4 * 4096 : 4096;  // per epilogue warp
  static constexpr int STAGING_BYTES = EW * WARP_BUF;
  static constexpr int EBARS = TMAE ? 2 * kEpiWarps : 0;
  static constexpr int BAR_BYTES = 8 * ((XF ? 3 : 2) * STAGES + 4 + EBARS) + 16;
  static constexpr int SMEM = 1024 + STAGES * STAGE_BYTES + STAGING_BYTES + BAR_BYTES;
  static_assert(SMEM <= 232448, "shared memory per CTA");
};


__device__ __forceinline__ void grid_decompose(int m, const PixGrid& g, int& n, int& i, int& j) {
  const int per = g.gh * g.gw;
  n = m / per;
  const int rem = m - n * per;
  i = rem / g.gw;
  j = rem - i * g.gw;
}

// Producer state of one work unit: everything that depends only on the tile
// is decomposed once, and the per-K-block coordinates advance incrementally
// (no integer divisions on the single issuing thread's critical path).
template <int BN>
struct Cursor {
  int kb;
  // A, im2col: input coordinates of the tile's first pixel; current tap / chunk
  int a_w, a_h, a_n, a_tap, a_c;
  // B, im2col (weight gradient): grid point of the K-block's first pixel and
  // the (tap, channel) of each 64-wide column chunk of the tile
  int b_n, b_i, b_j;
  int b_tap[BN / 64], b_c[BN / 64];
  // B, per-tap weight slices (data gradient): current tap / K chunk
  int b_t, b_k;

  __device__ __forceinline__ void init(const GemmParams& p, int m0, int n0, int kb0) {
    kb = kb0;
    if (p.a_mode == LD_IM2COL_K) {
      int n, i, j;
      grid_decompose(m0, p.ga, n, i, j);
      a_w = j * p.ga.step + p.ga.base_w;
      a_h = i * p.ga.step + p.ga.base_h;
      a_n = n;
      a_tap = kb0 / p.a_cpt;
      a_c = (kb0 - a_tap * p.a_cpt) * 64;
    }
    if (p.b_mode == LD_IM2COL_MN) {
      grid_decompose(kb0 * kBK, p.gb, b_n, b_i, b_j);
#pragma unroll
      for (int j = 0; j < BN / 64; ++j) {
        const int col = n0 + 64 * j;
        int tap = col / p.b_cin;
        int c0 = col - tap * p.b_cin;
        if (tap >= p.ntaps) {  // past the last tap: an all-out-of-bounds box (zeros)
          tap = 0;
          c0 = p.b_oob_c;
        }
        b_tap[j] = tap;
        b_c[j] = c0;
      }
    }
    if (p.b_mode == LD_TAP3D_MN) {
      b_t = kb0 / p.b_cpt;
      b_k = (kb0 - b_t * p.b_cpt) * 64;
    }
  }

  __device__ __forceinline__ void advance(const GemmParams& p) {
    ++kb;
    if (p.a_mode == LD_IM2COL_K) {
      a_c += 64;
      if (a_c == p.a_cpt * 64) {
        a_c = 0;
        ++a_tap;
      }
    }
    if (p.b_mode == LD_IM2COL_MN) {
      b_j += kBK;
      while (b_j >= p.gb.gw) {
        b_j -= p.gb.gw;
        if (++b_i == p.gb.gh) {
          b_i = 0;
          ++b_n;
        }
      }
    }
    if (p.b_mode == LD_TAP3D_MN) {
      b_k += 64;
      if (b_k == p.b_cpt * 64) {
        b_k = 0;
        ++b_t;
      }
    }
  }

  // the K-block's A and B boxes into stage (sa, sb), completing on bar
  __device__ __forceinline__ void load(const GemmParams& p, const CUtensorMap* ma, const CUtensorMap* mb,
                                       uint32_t sa, uint32_t sb, uint32_t bar, int m0, int n0) const {
    switch (p.a_mode) {
      case LD_TILED_K:
        tma_load_2d(sa, ma, bar, kb * kBK, m0);
        break;
      case LD_TILED_MN:
        tma_load_2d(sa, ma, bar, m0, kb * kBK);
        tma_load_2d(sa + 8192, ma, bar, m0 + 64, kb * kBK);
        break;
      case LD_IM2COL_K:
        tma_load_im2col_4d(sa, ma, bar, a_c, a_w, a_h, a_n, (uint16_t)p.tap_ds[a_tap],
                           (uint16_t)p.tap_dr[a_tap]);
        break;
      default:
        break;
    }
    switch (p.b_mode) {
      case LD_TILED_K:
        tma_load_2d(sb, mb, bar, kb * kBK, n0);
        break;
      case LD_TILED_MN:
#pragma unroll
        for (int j = 0; j < BN / 64; ++j) {
          tma_load_2d(sb + j * 8192, mb, bar, n0 + 64 * j, kb * kBK);
        }
        break;
      case LD_IM2COL_MN: {
        const int bw = b_j * p.gb.step + p.gb.base_w, bh = b_i * p.gb.step + p.gb.base_h;
#pragma unroll
        for (int j = 0; j < BN / 64; ++j) {
          tma_load_im2col_4d(sb + j * 8192, mb, bar, b_c[j], bw, bh, b_n, (uint16_t)p.tap_ds[b_tap[j]],
                             (uint16_t)p.tap_dr[b_tap[j]]);
        }
      } break;
      case LD_TAP3D_MN:
#pragma unroll
        for (int j = 0; j < BN / 64; ++j) {
          tma_load_3d(sb + j * 8192, mb, bar, n0 + 64 * j, p.tap_w[b_t], b_k);
        }
        break;
      default:
        break;
    }
  }
};

// Work unit u -> tile origin (m0, n0), split and K-block range (n tiles
// fastest, then M tiles, then splits).
__device__ __forceinline__ void unit_decode(const GemmParams& p, int u, int& m0, int& n0, int& split,
                                            int& kb0, int& kb1, int BN) {
  const int per = p.m_tiles * p.n_tiles;
  split = u / per;
  const int rem = u - split * per;
  const int mt = rem / p.n_tiles;
  m0 = mt * kBM;
  n0 = (rem - mt * p.n_tiles) * BN;
  if (p.nphase > 1) {  // the split index is the stride phase
    kb0 = p.ph_kb[split];
    kb1 = p.ph_kb[split + 1];
  } else {
    kb0 = split * p.kb_per_split;
    kb1 = min(p.num_kb, kb0 + p.kb_per_split);
  }
}

// Pixel row of GEMM row m of a stride phase (remap): grid point (n, i, j) ->
// (n, i * step + ph, j * step + pw).
__device__ __forceinline__ long long remap_row(const GemmParams& p, int m, int split) {
  const int per = p.rm_gh * p.rm_gw;
  const int n = m / per;
  const int rem = m - n * per;
  const int i = rem / p.rm_gw, j = rem - (rem / p.rm_gw) * p.rm_gw;
  const int ph = p.nphase > 1 ? p.ph_h[split] : p.rm_ph, pw = p.nphase > 1 ? p.ph_w[split] : p.rm_pw;
  return ((long long)n * p.rm_H + (long long)(i * p.rm_step + ph)) * p.rm_W + (j * p.rm_step + pw);
}

__device__ __forceinline__ uint16_t* out_row(const GemmParams& p, int m, int split) {
  long long row;
  if (p.out_mode == OUT_PARTIAL) {
    row = (long long)split * p.M + m;
  } else if (p.remap) {
    row = remap_row(p, m, split);
  } else {
    row = m;
  }
  return p.out + row * p.ldo;
}


// Register inputs of one 64-column chunk of the backward-statistics epilogue:
// the ReLU bits of row `lane` (all ones without a mask), the addend's mask
// bits of row `lane` (ADD; all ones without a mask) and the mean / invstd of
// channel pair (2 lane, 2 lane + 1).
struct ChunkIn {
  uint2 m, am;
  uint32_t mu2, is2;

  // row0: the tile's first row; prow >= 0: instead, the pixel row of row `lane`
  // (scattered rows of a stride phase), -1 past the tensor
  template <bool ADD>
  __device__ __forceinline__ void load(const GemmParams& p, long long row0, int col0, int lane,
                                       long long prow = -2) {
    const long long r = prow == -2 ? row0 + lane : prow;
    const bool in = prow == -2 ? r < p.M : prow >= 0;
    const long long mo = r * (p.N / 8) + col0 / 8;
    m = make_uint2(0xFFFFFFFFu, 0xFFFFFFFFu);
    if (p.bs_mask && in) m = __ldg(reinterpret_cast<const uint2*>(p.bs_mask + mo));
    am = make_uint2(0xFFFFFFFFu, 0xFFFFFFFFu);
    if (ADD && p.add_mask && in) am = __ldg(reinterpret_cast<const uint2*>(p.add_mask + mo));
    mu2 = __ldg(reinterpret_cast<const uint32_t*>(p.bs_mean + col0) + lane);
    is2 = __ldg(reinterpret_cast<const uint32_t*>(p.bs_invstd + col0) + lane);
  }
};

// Backward-statistics epilogue of one warp (BS, TMA stores): the warp's 32
// rows of each of its group's tiles (units u0, u0 + ustep, ...), 64 columns
// (a chunk) at a time.  Chunk q uses buffer b = q & 1 of the warp's four
// 128B-swizzled 32 x 64 tiles at wbuf: staging tile S[b] (the output; with ADD
// it first receives the addend) and input tile X[b] (the BatchNorm input x).
// The TMA loads of chunk q + 1 into buffer b ^ 1 are issued before chunk q is
// processed, completing on the warp's barrier wbar[b ^ 1]; its register inputs
// (ChunkIn) are loaded as far ahead.  With ADD the chunk's output is
// rn(result + addend) where the addend's mask bit is set (rn(result + 0)
// elsewhere), and the statistics are taken of that sum.
// REMAP (rows at the scattered pixels of a stride phase; no ADD): every lane
// fetches 16-byte pieces of x's rows with cp.async into the swizzled X[b]
// (the barrier then expects 32 arrivals), and the chunk leaves S[b] by plain
// stores of whole 128-byte row segments instead of a TMA store.
template <int BN, bool ADD, bool REMAP>
__device__ __forceinline__ void epilogue_bs(const GemmParams& p, const CUtensorMap* mapC, const CUtensorMap* mapX,
                                            const CUtensorMap* mapD, uint8_t* wbuf, uint64_t* wbar,
                                            uint64_t* tfull, uint64_t* tempty, uint32_t tmem_base, int acc, int sub,
                                            int lane, int u0, int ustep, int total, uint64_t lim,
                                            volatile int* abort_flag, EpiStats& stats) {
  static_assert(!(ADD && REMAP), "the addend's rows are in pixel order");
  if (u0 >= total) return;
  const uint32_t S0 = smem_u32(wbuf), X0 = S0 + 2 * 4096;
  const uint32_t B0 = smem_u32(wbar);
  const uint32_t tx = ADD ? 2 * 4096 : 4096;
  const int rq = lane >> 3, cj = lane & 7;  // REMAP: rows rq + 4 i, 16-byte column cj
  // lane 0: the chunk index whose loads are in flight in each buffer (-1: none)
  int pend[2] = {-1, -1};
  auto issue = [&](int b, int row0, int col0, int q) {
    mbar_arrive_expect_tx(B0 + 8 * b, tx);
    tma_load_2d(X0 + b * 4096, mapX, B0 + 8 * b, col0, row0);
    if (ADD) tma_load_2d(S0 + b * 4096, mapD, B0 + 8 * b, col0, row0);
    pend[b] = q;
  };
  // REMAP, all lanes: rows of the chunk whose row `lane` is at pixel row prow (-1: past the tensor)
  auto issue_rows = [&](int b, long long prow, int col0, int q) {
    const uint32_t xb = X0 + b * 4096;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int rr = rq + 4 * i;
      const long long pr = __shfl_sync(0xffffffffu, prow, rr);
      if (pr >= 0) cp_async_16(xb + rr * 128 + ((cj ^ (rr & 7)) << 4), p.bs_x + pr * p.ldo + col0 + 8 * cj);
    }
    cp_async_mbar_arrive_noinc(B0 + 8 * b);
    if (lane == 0) pend[b] = q;
  };
  // REMAP: the pixel row of row `lane` of the tile at m (-1 past the tensor)
  auto pixel_row = [&](int m, int sp) -> long long {
    const int mr = m + sub * 32 + lane;
    return mr < p.M ? remap_row(p, mr, sp) : -1ll;
  };
  int u = u0, m0, n0, split, kb0, kb1;
  unit_decode(p, u, m0, n0, split, kb0, kb1, BN);
  int c = 0;
  long long prow = 0, prow2 = 0;
  if constexpr (REMAP) {
    prow = pixel_row(m0, split);
    issue_rows(0, prow, n0, 0);
  } else if (lane == 0) {
    issue(0, m0 + sub * 32, n0, 0);
  }
  ChunkIn cur, nxt;
  cur.load<ADD>(p, (long long)(m0 + sub * 32), n0, lane, REMAP ? prow : -2);
  uint32_t acc_phase = 0, tbase = 0;
  int nv = 0;
  for (int q = 0;; ++q) {
    if (c == 0) {  // a new tile: wait for its accumulator
      if (__any_sync(0xffffffffu, *abort_flag != 0)) break;
      const bool got = mbar_wait(smem_u32(&tfull[acc]), acc_phase, lim);
      if (!__all_sync(0xffffffffu, got)) {
        if (lane == 0) record_timeout(p, abort_flag);
        break;
      }
      tc_fence_after();
      tbase = tmem_base + ((uint32_t)(sub * 32) << 16) + (uint32_t)(acc * BN);
      nv = min(32, max(0, p.M - (m0 + sub * 32)));
    }
    const int b = q & 1;
    // the next chunk: this tile's next 64 columns, else the group's next tile
    int u2 = u, c2 = c + 64, m2 = m0, n2 = n0;
    const bool last = c2 >= BN || n0 + c2 >= p.N;  // the tile's last chunk
    if (last) {
      u2 = u + ustep;
      c2 = 0;
      if (u2 < total) unit_decode(p, u2, m2, n2, split, kb0, kb1, BN);
    }
    const bool more = u2 < total;
    if (more) {
      __syncwarp();  // every lane is done reading buffer b ^ 1 (chunk q - 1)
      if constexpr (REMAP) {
        prow2 = last ? pixel_row(m2, split) : prow;
        issue_rows(b ^ 1, prow2, n2 + c2, q + 1);
      } else if (lane == 0) {
        bulk_wait_read0();         // chunk q - 1's store has read S[b ^ 1]
        fence_proxy_async_smem();  // the warp's reads of X[b ^ 1] before the copy's writes
        issue(b ^ 1, m2 + sub * 32, n2 + c2, q + 1);
      }
      nxt.load<ADD>(p, (long long)(m2 + sub * 32), n2 + c2, lane, REMAP ? prow2 : -2);
    }
    uint32_t r[64];
    tmem_ld16(tbase + c, r);
    tmem_ld16(tbase + c + 16, r + 16);
    tmem_ld16(tbase + c + 32, r + 32);
    tmem_ld16(tbase + c + 48, r + 48);
    tmem_ld_wait();
    if (p.d_f32) f32_to_f16_lo<64>(r);  // FP32 accumulator: one rounding to FP16
    if (last) {  // accumulator fully read: hand TMEM back
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&tempty[acc]));
    }
    const bool ok = mbar_wait(B0 + 8 * b, (uint32_t)(q >> 1) & 1u, lim);
    if (!__all_sync(0xffffffffu, ok)) {
      if (lane == 0) record_timeout(p, abort_flag);
      break;
    }
    if (lane == 0) pend[b] = -1;
    const uint32_t S = S0 + b * 4096, X = X0 + b * 4096;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      uint4 v;
      v.x = pack_lo(r[j * 8 + 0], r[j * 8 + 1]);
      v.y = pack_lo(r[j * 8 + 2], r[j * 8 + 3]);
      v.z = pack_lo(r[j * 8 + 4], r[j * 8 + 5]);
      v.w = pack_lo(r[j * 8 + 6], r[j * 8 + 7]);
      const uint32_t addr = S + lane * 128 + ((j ^ (lane & 7)) << 4);
      if (ADD) {
        uint4 a;
        ld_shared_v4(addr, a);
        const uint32_t bits = ((j < 4 ? cur.am.x : cur.am.y) >> (8 * (j & 3))) & 0xFFu;
        uint32_t mk[4];
#pragma unroll
        for (int k = 0; k < 4; ++k)
          mk[k] = (((bits >> (2 * k)) & 1u) ? 0x0000FFFFu : 0u) | (((bits >> (2 * k + 1)) & 1u) ? 0xFFFF0000u : 0u);
        v.x = hadd2_rn(v.x, a.x & mk[0]);
        v.y = hadd2_rn(v.y, a.y & mk[1]);
        v.z = hadd2_rn(v.z, a.z & mk[2]);
        v.w = hadd2_rn(v.w, a.w & mk[3]);
      }
      st_shared_v4(addr, v);
    }
    if constexpr (REMAP) {
      __syncwarp();
      const int n = n0 + c + 8 * cj;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int rr = rq + 4 * i;
        const long long pr = __shfl_sync(0xffffffffu, prow, rr);
        uint4 v;
        ld_shared_v4(S + rr * 128 + ((cj ^ (rr & 7)) << 4), v);
        if (pr >= 0 && n + 8 <= p.N) *reinterpret_cast<uint4*>(p.out + pr * p.ldo + n) = v;
      }
    } else {
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        tma_store_2d(mapC, S, n0 + c, m0 + sub * 32);
        bulk_commit();
      }
    }
    if (p.st_mean && nv > 0) stats.leaf_bwd_tile(c / 64, S, X, lane, nv, cur.m, cur.mu2, cur.is2);
    if (last) {
      if (p.st_mean && nv > 0) stats.end_tile(nv);
      acc_phase ^= 1;
    }
    if (!more) break;
    cur = nxt;
    prow = prow2;
    u = u2;
    c = c2;
    m0 = m2;
    n0 = n2;
  }
  // after an abort: let the loads still in flight land before shared memory is released
  if (lane == 0)
    for (int b = 0; b < 2; ++b)
      if (pend[b] >= 0) mbar_wait(B0 + 8 * b, (uint32_t)(pend[b] >> 1) & 1u, 1000000000ull);
}

// ---------------------------------------------------------------------------
// BatchNorm in the operand path (GemmParams::xf_*).  An operand stage is
// made of 128-byte rows -- one pixel's 64 channels, 128B-swizzled: channel
// chunk g of row r sits in 16-byte slot g ^ (r & 7) -- and is replaced in
// place by the BatchNorm's output, with the apply pass's op sequence.  Each
// transform thread owns one slot column of rows congruent mod 8 (so a single
// channel chunk and one set of per-channel parameters), loads all its rows
// before computing and stores after, and holds the parameters in registers,
// loaded ahead of use.
//   A (K-major, 128 pixel rows, the 64 channels of K-block kb): thread t takes
//     slot t & 7 of rows t / 8 + 32 i (4 rows).
//   B (MN-major, BN / 64 atoms of 64 pixel rows, atom j = channels n0 + 64 j):
//     tpa = 256 / 2^ceil(log2(BN / 64)) threads per atom; thread t takes atom
//     t / tpa, slot t & 7 of rows (t % tpa) / 8 + (tpa / 8) i.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t xf_pair(uint32_t x, uint32_t mu, uint32_t is, uint32_t ga, uint32_t be,
                                            uint32_t ps) {
  const uint32_t xh = hmul2_rn(hsub2_rn(x, mu), is);  // Eq. 1
  return hmul2_rn(hadd2_rn(hmul2_rn(ga, xh), be), ps);  // Eq. 2, then x post_scale (Sec. 4.2)
}
// bit 15 of each 16-bit lane set where the lane is > 0 and not NaN: magnitude
// m = h & 0x7FFF non-zero (m + 0x7FFF carries into bit 15), at most 0x7C00
// (m + 0x3FF does not), sign clear.  No carry crosses a lane.
__device__ __forceinline__ uint32_t pos15(uint32_t h) {
  const uint32_t m = h & 0x7FFF7FFFu;
  return (m + 0x7FFF7FFFu) & ~((m + 0x03FF03FFu) | h) & 0x80008000u;
}

struct XfParams {
  uint4 mu, is, ga, be;
  __device__ __forceinline__ void load(const GemmParams& p, int c) {
    if (c < p.xf_C) {
      mu = __ldg(reinterpret_cast<const uint4*>(p.xf_mean + c));
      is = __ldg(reinterpret_cast<const uint4*>(p.xf_invstd + c));
      ga = __ldg(reinterpret_cast<const uint4*>(p.xf_gamma + c));
      be = __ldg(reinterpret_cast<const uint4*>(p.xf_beta + c));
    }
  }
};

// Transform `n` rows (row i at smem address a0 + i * astep, pixel pix0 + i *
// pstep) of one slot column holding channels c .. c + 7.
template <int MAXR>
__device__ __forceinline__ void xf_rows(const GemmParams& p, const XfParams& q, uint32_t a0, uint32_t astep, int n,
                                        long long pix0, long long pstep, int c, uint8_t* mask_out) {
  const bool cok = c < p.xf_C;
  const uint32_t ps = (uint32_t)p.xf_scale | ((uint32_t)p.xf_scale << 16);
  uint4 v[MAXR];
#pragma unroll
  for (int i = 0; i < MAXR; ++i)
    if (i < n) ld_shared_v4(a0 + (uint32_t)i * astep, v[i]);
  const long long cpr = p.xf_C / 8;  // mask bytes per pixel row
#pragma unroll
  for (int i = 0; i < MAXR; ++i) {
    if (i >= n) break;
    const long long pix = pix0 + (long long)i * pstep;
    uint4 z = make_uint4(0, 0, 0, 0);
    if (cok && pix < p.xf_rows) {
      z.x = xf_pair(v[i].x, q.mu.x, q.is.x, q.ga.x, q.be.x, ps);
      z.y = xf_pair(v[i].y, q.mu.y, q.is.y, q.ga.y, q.be.y, ps);
      z.z = xf_pair(v[i].z, q.mu.z, q.is.z, q.ga.z, q.be.z, ps);
      z.w = xf_pair(v[i].w, q.mu.w, q.is.w, q.ga.w, q.be.w, ps);
      if (p.xf_relu) {
        const uint32_t k0 = pos15(z.x), k1 = pos15(z.y), k2 = pos15(z.z), k3 = pos15(z.w);
        z = make_uint4(z.x & ((k0 >> 15) * 0xFFFFu), z.y & ((k1 >> 15) * 0xFFFFu), z.z & ((k2 >> 15) * 0xFFFFu),
                       z.w & ((k3 >> 15) * 0xFFFFu));
        if (mask_out) {
          // lane 2k's decision (bit 15 of word k) -> bit 2k, lane 2k+1's (bit 31) -> bit 2k+1
          const uint32_t b = (k0 >> 15 & 1u) | (k0 >> 30 & 2u) | (k1 >> 13 & 4u) | (k1 >> 28 & 8u) |
                             (k2 >> 11 & 16u) | (k2 >> 26 & 32u) | (k3 >> 9 & 64u) | (k3 >> 24 & 128u);
          mask_out[pix * cpr + c / 8] = (uint8_t)b;
        }
      }
    }
    v[i] = z;
  }
#pragma unroll
  for (int i = 0; i < MAXR; ++i)
    if (i < n) st_shared_v4(a0 + (uint32_t)i * astep, v[i]);
}

// EPI: the epilogue's kind, each a separate instantiation so that the others
// do not carry its registers or give up its pipeline stages --
//   EPI_PLAIN: stores (forward statistics optional);
//   EPI_BS: BatchNorm backward statistics (GemmParams::bs_x), inputs loaded
//     into registers (for long reductions, which need every pipeline stage);
//   EPI_BS_TMA: the same statistics from TMA-fed tiles (epilogue_bs; for short
//     reductions, whose epilogue is the bound);
//   EPI_BS_ADD: EPI_BS_TMA plus the addend (GemmParams::add_src).
//   EPI_BS_REMAP: EPI_BS_TMA for the scattered rows of a stride phase (x by
//     cp.async, the output by plain stores).
// XF (with EPI_PLAIN): BatchNorm in the operand path (GemmParams::xf_*):
// eight more warps transform each stage between the TMA's arrival (full) and
// the MMAs (xready), see xf_rows.
// WE (with EPI_PLAIN, TMA stores): the wide epilogue, warps 2-17 in four
// groups: group g drains accumulator g & 1, columns of half g >> 1.
template <int BN, int EPI, bool XF = false, bool WE = false>
__global__ void __launch_bounds__(XF ? kGemmThreadsXf : (WE ? kGemmThreadsWide : kGemmThreads), 1)
    k_gemm(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB,
           const __grid_constant__ CUtensorMap mapC, const __grid_constant__ CUtensorMap mapX,
           const __grid_constant__ CUtensorMap mapD, const __grid_constant__ GemmParams p) {
  constexpr bool BS = EPI != EPI_PLAIN, ADD = EPI == EPI_BS_ADD, REMAP = EPI == EPI_BS_REMAP;
  constexpr bool TMAE = EPI == EPI_BS_TMA || ADD || REMAP;
  static_assert(!WE || (EPI == EPI_PLAIN && !XF && BN % 128 == 0), "the wide epilogue: plain, BN 128 or 256");
  using Cfg = GemmCfg<BN, TMAE, XF, WE>;
  constexpr int CS = WE ? 2 : 1;  // column halves per tile
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* staging = smem + Cfg::STAGES * Cfg::STAGE_BYTES;  // 1024-aligned, 2 x 4 KB per epilogue warp
  uint64_t* bars = reinterpret_cast<uint64_t*>(staging + Cfg::STAGING_BYTES);
  uint64_t* full = bars;
  uint64_t* empty = bars + Cfg::STAGES;
  uint64_t* tfull = bars + 2 * Cfg::STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* ebar = tempty + 2;  // TMAE: per epilogue warp, one transaction barrier per input buffer
  uint64_t* xready = ebar + Cfg::EBARS;  // XF: the stage has been transformed
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(xready + (XF ? Cfg::STAGES : 0));
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < Cfg::STAGES; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&tfull[a]), 1);
      mbar_init(smem_u32(&tempty[a]), 4 * CS);  // every warp that drains the accumulator arrives
    }
    // (a stride phase's x rows arrive by every lane's cp.async: 32 arrivals)
    for (int b = 0; b < Cfg::EBARS; ++b) mbar_init(smem_u32(&ebar[b]), REMAP ? 32 : 1);
    if (XF)
      for (int s = 0; s < Cfg::STAGES; ++s) mbar_init(smem_u32(&xready[s]), kXfWarps);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&mapA);
    tma_prefetch_desc(&mapB);
    if (p.tma_store) tma_prefetch_desc(&mapC);
    if (TMAE) tma_prefetch_desc(&mapX);
    if (ADD) tma_prefetch_desc(&mapD);
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
  // work enumeration: CTA cid takes units cid, cid + ncl, ...
  const int cid = (int)blockIdx.x;
  const int ncl = (int)gridDim.x;
  const int total = p.m_tiles * p.n_tiles * p.splits;
  const uint64_t lim = p.wait_limit_ns;

  if (warp == 0) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued = 0;  // stages loaded so far (for the drain below)
      for (int u = cid; u < total && !*abort_flag; u += ncl) {
        int m0, n0, split, kb0, kb1;
        unit_decode(p, u, m0, n0, split, kb0, kb1, BN);
        Cursor<BN> cur;
        cur.init(p, m0, n0, kb0);
        for (int kb = kb0; kb < kb1; ++kb, cur.advance(p)) {
          if (!mbar_wait(smem_u32(&empty[stage]), phase ^ 1, lim)) {
            record_timeout(p, abort_flag);
            break;
          }
          const uint32_t sa = smem_u32(smem + stage * Cfg::STAGE_BYTES);
          const uint32_t fb = smem_u32(&full[stage]);
          mbar_arrive_expect_tx(fb, Cfg::STAGE_BYTES);
          cur.load(p, &mapA, &mapB, sa, sa + Cfg::A_BYTES, fb, m0, n0);
          ++issued;
          if (++stage == Cfg::STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (*abort_flag) {
        // Another role gave up: let the copies this thread started land before
        // the CTA's shared memory is released (each wait bounded on its own).
        const uint32_t n = issued < (uint32_t)Cfg::STAGES ? issued : (uint32_t)Cfg::STAGES;
        int s = stage;
        uint32_t ph = phase;
        for (uint32_t i = 0; i < n; ++i) {
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
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      // base descriptors (address field 0) and K-step strides in 16-byte units:
      // a step's descriptor is one add away
      const uint64_t adesc0 = smem_desc(0, p.a_lbo, p.a_sbo, 2);
      const uint64_t bdesc0 = smem_desc(0, p.b_lbo, p.b_sbo, 2);
      const uint32_t ak16 = (uint32_t)p.a_kstep >> 4, bk16 = (uint32_t)p.b_kstep >> 4;
      for (int u = cid; u < total && !*abort_flag; u += ncl) {
        int m0, n0, split, kb0, kb1;
        unit_decode(p, u, m0, n0, split, kb0, kb1, BN);
        if (!mbar_wait(smem_u32(&tempty[acc]), acc_phase ^ 1, lim)) {
          record_timeout(p, abort_flag);
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
        bool ok = true;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(smem_u32(XF ? &xready[stage] : &full[stage]), phase, lim)) {
            record_timeout(p, abort_flag);
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa16 = desc_addr16(smem_u32(smem + stage * Cfg::STAGE_BYTES));
          const uint64_t ab = adesc0 + sa16, bb = bdesc0 + sa16 + (Cfg::A_BYTES >> 4);
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk)
            tc_mma_f16(d_tmem, ab + kk * ak16, bb + kk * bk16, p.idesc, (kb > kb0 || kk > 0) ? 1u : 0u);
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
    }
  } else if (XF && warp >= kXfWarp0) {
    // transform warps: each stage, once the TMA has landed, into the BatchNorm's output
    const int xt = threadIdx.x - 32 * kXfWarp0;  // 0 .. 255
    const int slot = xt & 7;
    // B: atoms of this stage, threads per atom (a power of two), this thread's atom and rows
    constexpr int kAtoms = BN / 64;
    constexpr int kTpa = kAtoms == 1 ? 256 : (kAtoms == 2 ? 128 : 64);
    const int bj = xt / kTpa, btt = xt % kTpa, brow0 = btt >> 3;
    const bool bact = bj < kAtoms;
    const int arow0 = xt >> 3;  // A: rows arow0 + 32 i
    const int ag = slot ^ (arow0 & 7), bg = slot ^ (brow0 & 7);
    int stage = 0;
    uint32_t phase = 0;
    XfParams q;
    bool have_next = false;  // A: q already holds the parameters of the next K-block
    for (int u = cid; u < total; u += ncl) {
      if (__any_sync(0xffffffffu, *abort_flag != 0)) break;
      int m0, n0, split, kb0, kb1;
      unit_decode(p, u, m0, n0, split, kb0, kb1, BN);
      if (p.xf_operand == 2) {
        q.load(p, n0 + 64 * bj + 8 * bg);  // constant over the unit's K-blocks
      } else if (!have_next) {
        q.load(p, kb0 * kBK + 8 * ag);
      }
      bool ok = true;
      for (int kb = kb0; kb < kb1; ++kb) {
        const bool got = mbar_wait(smem_u32(&full[stage]), phase, lim);
        if (!__all_sync(0xffffffffu, got)) {
          if (lane == 0) record_timeout(p, abort_flag);
          ok = false;
          break;
        }
        const uint32_t sa = smem_u32(smem + stage * Cfg::STAGE_BYTES);
        if (p.xf_operand == 1) {
          const XfParams cur = q;
          // the next K-block's parameters, in flight while this one is transformed
          int nkb = kb + 1;
          if (nkb >= kb1) {
            int u2 = u + ncl, mm, nn, ss, k0, k1;
            nkb = -1;
            if (u2 < total) {
              unit_decode(p, u2, mm, nn, ss, k0, k1, BN);
              nkb = k0;
            }
          }
          have_next = nkb >= 0;
          if (have_next) q.load(p, nkb * kBK + 8 * ag);
          const uint32_t a0 = sa + (uint32_t)arow0 * 128u + (uint32_t)slot * 16u;
          xf_rows<kBM / 32>(p, cur, a0, 32u * 128u, kBM / 32, (long long)m0 + arow0, 32, kb * kBK + 8 * ag,
                            (p.xf_mask != nullptr && n0 == 0) ? p.xf_mask : nullptr);
        } else if (bact) {
          const uint32_t a0 = sa + Cfg::A_BYTES + (uint32_t)bj * 8192u + (uint32_t)brow0 * 128u + (uint32_t)slot * 16u;
          xf_rows<512 / kTpa>(p, q, a0, (uint32_t)(kTpa / 8) * 128u, 512 / kTpa, (long long)kb * kBK + brow0,
                              kTpa / 8, n0 + 64 * bj + 8 * bg, nullptr);
        }
        fence_proxy_async_smem();  // the transformed tile, before the tensor core reads it
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&xready[stage]));
        if (++stage == Cfg::STAGES) {
          stage = 0;
          phase ^= 1;
        }
      }
      if (!ok) break;
    }
  } else {
    // epilogue warps 2..9 (2..17 with WE) -> TMEM sub-partitions 2, 3, 0, 1, ...; group grp
    // drains accumulator grp & 1, columns [c_begin, c_end) (the whole tile, or half of it)
    const int e = warp - 2, grp = e >> 2, sub = warp & 3;
    const int acc = grp & 1;
    const int c_begin = WE ? (grp >> 1) * (BN / CS) : 0, c_end = c_begin + BN / CS;
    uint32_t acc_phase = 0;
    const uint32_t stg = smem_u32(staging) + (uint32_t)(e * Cfg::WARP_BUF);
    EpiStats stats;
    stats.init();
    // tcgen05.ld is warp-collective: every exit decision below is warp-uniform
    if constexpr (TMAE)  // (rows in pixel order with TMA stores, or the scattered rows of a stride phase)
      epilogue_bs<BN, ADD, REMAP>(p, &mapC, &mapX, &mapD, staging + e * Cfg::WARP_BUF, ebar + 2 * e, tfull, tempty,
                                  tmem_base, acc, sub, lane, cid + grp * ncl, 2 * ncl, total, lim, abort_flag, stats);
    const bool bstats = BS && p.st_mean && p.bs_x && p.tma_store;
    BwdIn bin;
    for (int u = cid + acc * ncl; u < total && !TMAE; u += 2 * ncl) {
      if (__any_sync(0xffffffffu, *abort_flag != 0)) break;
      int m0, n0, split, kb0, kb1;
      unit_decode(p, u, m0, n0, split, kb0, kb1, BN);
      if (bstats) {  // the first chunk's inputs, loaded while the accumulator is computed
        const int nv0 = min(32, max(0, p.M - (m0 + sub * 32)));
        if (nv0 > 0) bin.load(p, (long long)(m0 + sub * 32), n0, nv0, lane);
      }
      const bool got = mbar_wait(smem_u32(&tfull[acc]), acc_phase, lim);
      if (!__all_sync(0xffffffffu, got)) {
        if (lane == 0) record_timeout(p, abort_flag);
        break;
      }
      tc_fence_after();
      const uint32_t tbase = tmem_base + ((uint32_t)(sub * 32) << 16) + (uint32_t)(acc * BN);
      if (p.tma_store) {
        // valid rows of this warp (a prefix of its 32) for the fused statistics
        const int nv = min(32, max(0, p.M - (m0 + sub * 32)));
        // 64-column chunks: TMEM -> registers -> 128B-swizzled staging -> TMA store
#pragma unroll 1
        for (int c = c_begin; c < c_end; c += 64) {
          uint32_t r[64];
          tmem_ld16(tbase + c, r);
          tmem_ld16(tbase + c + 16, r + 16);
          tmem_ld16(tbase + c + 32, r + 32);
          tmem_ld16(tbase + c + 48, r + 48);
          tmem_ld_wait();
          if (p.d_f32) f32_to_f16_lo<64>(r);  // FP32 accumulator: one rounding to FP16
          if (c + 64 >= c_end) {  // this warp's columns fully read: hand TMEM back before the stores
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
          if (lane == 0) {
            if (p.out_mode == OUT_PARTIAL)
              tma_store_3d(&mapC, stg, n0 + c, m0 + sub * 32, split);
            else if (p.out_mode == OUT_ACCUM)
              tma_reduce_add_2d(&mapC, stg, n0 + c, m0 + sub * 32);
            else
              tma_store_2d(&mapC, stg, n0 + c, m0 + sub * 32);
            bulk_commit();
          }
          if (p.st_mean && nv > 0 && n0 + c < p.N) {
            if (BS) {
              stats.leaf_bwd(c / 64, stg, lane, nv, bin);
              if (c + 64 < BN && n0 + c + 64 < p.N) bin.load(p, (long long)(m0 + sub * 32), n0 + c + 64, nv, lane);
            } else {
              stats.leaf(c / 64, stg, lane, nv);
            }
          }
        }
        if (p.st_mean && nv > 0) stats.end_tile(nv);
        acc_phase ^= 1;
        continue;
      }
      if constexpr (!XF) {  // (the operand-transform variants never take remapped rows)
        // Rows remapped to strided positions (a stride phase): each 64-column
        // chunk goes through the warp's 128B-swizzled staging tile, then lane l
        // moves 16 bytes (columns 8 (l % 8) ..) of rows l / 8 + 4 i, i < 8: a
        // warp instruction writes four whole 128-byte row segments.
        const int rq = lane >> 3, cj = lane & 7;
        uint16_t* orow[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int m = m0 + sub * 32 + rq + 4 * i;
          orow[i] = m < p.M ? out_row(p, m, split) : nullptr;
        }
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
          __syncwarp();  // every lane is done reading the previous chunk from the staging tile
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            uint4 v;
            v.x = pack_lo(r[j * 8 + 0], r[j * 8 + 1]);
            v.y = pack_lo(r[j * 8 + 2], r[j * 8 + 3]);
            v.z = pack_lo(r[j * 8 + 4], r[j * 8 + 5]);
            v.w = pack_lo(r[j * 8 + 6], r[j * 8 + 7]);
            st_shared_v4(stg + lane * 128 + ((j ^ (lane & 7)) << 4), v);
          }
          __syncwarp();
          const int n = n0 + c + 8 * cj;
          if (n + 8 <= p.N) {
            uint4 v[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              const int rr = rq + 4 * i;
              ld_shared_v4(stg + rr * 128 + ((cj ^ (rr & 7)) << 4), v[i]);
            }
            if (p.out_mode == OUT_ACCUM) {
              uint4 o[8];
#pragma unroll
              for (int i = 0; i < 8; ++i)
                o[i] = orow[i] ? *reinterpret_cast<const uint4*>(orow[i] + n) : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
              for (int i = 0; i < 8; ++i) {
                v[i].x = hadd2_rn(o[i].x, v[i].x);
                v[i].y = hadd2_rn(o[i].y, v[i].y);
                v[i].z = hadd2_rn(o[i].z, v[i].z);
                v[i].w = hadd2_rn(o[i].w, v[i].w);
              }
            }
#pragma unroll
            for (int i = 0; i < 8; ++i)
              if (orow[i]) *reinterpret_cast<uint4*>(orow[i] + n) = v[i];
          }
        }
      }
      acc_phase ^= 1;
    }
    if (p.tma_store && lane == 0) bulk_wait0();
    if (p.st_mean) {
      // this CTA's tiles all have n-tile cid % n_tiles (the grid is a multiple of n_tiles);
      // slot cid / n_tiles
      const int n0 = (cid % p.n_tiles) * BN;
      const int nch = min(BN, p.N - n0) / 64;
      const int slot = cid / p.n_tiles;
      if (BS)
        stats.write_cta_bwd(p, staging, e, slot, n0, nch, lane, p.bs_levels);
      else
        stats.write_cta(p, staging, e, slot, n0, nch, lane, cid % p.n_tiles == 0, Cfg::EW, BN / 64 / CS);
      if (blockIdx.x == 0 && e == 0 && lane == 0) {
        p.st_hdr[0] = ncl / p.n_tiles;
        p.st_hdr[1] = 5 + p.bs_levels + 3;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, Cfg::TMEM_COLS);
  }
}

int gemm_smem_bytes(int BN) {
  switch (BN) {
    case 64: return GemmCfg<64>::SMEM;
    case 128: return GemmCfg<128>::SMEM;
    case 192: return GemmCfg<192>::SMEM;
    case 256: return GemmCfg<256>::SMEM;
    default: return -1;
  }
}

template <int BN, int EPI = EPI_PLAIN, bool XF = false, bool WE = false>
static cudaError_t set_smem_attr() {
  static bool attr_set[64] = {false};  // per device ordinal
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 64 && !attr_set[dev]) {
    cudaError_t e = cudaFuncSetAttribute(k_gemm<BN, EPI, XF, WE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         GemmCfg<BN, EPI == EPI_BS_TMA || EPI == EPI_BS_ADD || EPI == EPI_BS_REMAP, XF, WE>::SMEM);
    if (e != cudaSuccess) return e;
    attr_set[dev] = true;
  }
  return cudaSuccess;
}

template <int BN, int EPI, bool XF = false, bool WE = false>
static cudaError_t launch_variant(const CUtensorMap& mA, const CUtensorMap& mB, const CUtensorMap& mC,
                                  const CUtensorMap& mX, const CUtensorMap& mD, const GemmParams& p, int grid,
                                  cudaStream_t s) {
  cudaError_t e = set_smem_attr<BN, EPI, XF, WE>();
  if (e != cudaSuccess) return e;
  constexpr int smem = GemmCfg<BN, EPI == EPI_BS_TMA || EPI == EPI_BS_ADD || EPI == EPI_BS_REMAP, XF, WE>::SMEM;
  launch_pdl(k_gemm<BN, EPI, XF, WE>, dim3(grid), dim3(XF ? kGemmThreadsXf : (WE ? kGemmThreadsWide : kGemmThreads)),
             smem, s, mA, mB, mC, mX, mD, p);
  return counted_launches(1);
}

template <int BN>
static cudaError_t launch_bn_t(const CUtensorMap& mA, const CUtensorMap& mB, const CUtensorMap& mC,
                               const CUtensorMap& mX, const CUtensorMap& mD, const GemmParams& p, int grid,
                               cudaStream_t s) {
  const int epi = gemm_epilogue(p);
  if (epi != EPI_PLAIN && p.out_mode != OUT_STORE) return cudaErrorInvalidValue;
  if (epi != EPI_PLAIN && !p.tma_store && !(epi == EPI_BS_REMAP && p.remap)) return cudaErrorInvalidValue;
  if (p.xf_operand) {
    if (epi != EPI_PLAIN) return cudaErrorInvalidValue;
    return launch_variant<BN, EPI_PLAIN, true>(mA, mB, mC, mX, mD, p, grid, s);
  }
  // the shortest reductions (one or two K-blocks per tile) with a plain
  // epilogue: the wide epilogue, whose 16 warps drain a tile's two column
  // halves at once -- there the epilogue is the bound (56x56 64->256 forward
  // with statistics 117 -> 103 us); from four K-blocks on, the pipeline stages
  // it gives up cost more (14x14 256->1024 forward 42.2 -> 44.0 us)
  if constexpr (BN == 128 || BN == 256)
    if (epi == EPI_PLAIN && p.tma_store && p.kb_per_split <= 2)
      return launch_variant<BN, EPI_PLAIN, false, true>(mA, mB, mC, mX, mD, p, grid, s);
  switch (epi) {
    case EPI_PLAIN: return launch_variant<BN, EPI_PLAIN>(mA, mB, mC, mX, mD, p, grid, s);
    case EPI_BS: return launch_variant<BN, EPI_BS>(mA, mB, mC, mX, mD, p, grid, s);
    case EPI_BS_TMA: return launch_variant<BN, EPI_BS_TMA>(mA, mB, mC, mX, mD, p, grid, s);
    case EPI_BS_ADD: return launch_variant<BN, EPI_BS_ADD>(mA, mB, mC, mX, mD, p, grid, s);
    case EPI_BS_REMAP: return launch_variant<BN, EPI_BS_REMAP>(mA, mB, mC, mX, mD, p, grid, s);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_gemm(int BN, const CUtensorMap& mA, const CUtensorMap& mB, const CUtensorMap& mC,
                        const GemmParams& p, int grid, cudaStream_t s, const CUtensorMap* mX,
                        const CUtensorMap* mD) {
  // the BatchNorm-input and addend maps (unused without backward statistics)
  const CUtensorMap& x = mX ? *mX : mC;
  const CUtensorMap& d = mD ? *mD : x;
  switch (BN) {
    case 64: return launch_bn_t<64>(mA, mB, mC, x, d, p, grid, s);
    case 128: return launch_bn_t<128>(mA, mB, mC, x, d, p, grid, s);
    case 192: return launch_bn_t<192>(mA, mB, mC, x, d, p, grid, s);
    case 256: return launch_bn_t<256>(mA, mB, mC, x, d, p, grid, s);
    default: return cudaErrorInvalidValue;
  }
}


// ---------------------------------------------------------------------------
// Halo engine: stride-1 convolution with 64 outputs read from a padded pixel
// grid.  GEMM rows are the pixels of a grid whose image rows are ws columns
// wide (ws = 32, 64 or 128, at least the output width plus the filter width
// minus one), so a 128-row tile is 128/ws whole output rows.  One TMA box
// brings the input rows and columns the tile's taps touch (zeros outside the
// image), one pixel per swizzled row of cb bytes; tap (dr, ds) is then the
// 128-row window that starts dr*ws + ds pixels into the box.  The swizzle is
// a function of the absolute shared-memory address, so a descriptor whose
// start moves by whole rows reads exactly that window (checked on the GPU for
// 128-byte rows: rows m + o for offsets o = 1, 2, 3, 8, 9 with base offset 0).
// The input is thus read once per tile instead of once per tap, and the taps'
// weight slices stay in shared memory for the whole launch.  Two uses:
//   - 3x3 / stride 1 / pad 1, 64 -> 64 channels (forward, or the data
//     gradient as a convolution of dy with the flipped filter): cb = 128,
//     128-byte swizzle, box rows i0-1 .. i0+128/ws, columns -1 .. ws-2; one
//     N = 192 MMA per filter row and K step (three taps' slices against one
//     window, recombined by row shifts in the epilogue: halo3_combine);
//   - the 7x7 / stride 2 / pad 3 stem after a 2x2 space-to-depth of its
//     three-channel input: a 4x4 / stride 1 / unpadded convolution over 16
//     channels (12 real), cb = 32, 32-byte swizzle, one K = 16 MMA per tap.
// Columns j >= Q of the padded grid are computed and then dropped by the 3-D
// TMA store, which clips at Q.
// Same roles and bounded waits as k_gemm.
// ---------------------------------------------------------------------------
struct HaloCfg {
  static constexpr int B_BYTES = 9 * 64 * kBK * 2;  // resident: 9 taps x 64 x 64, or 16 x 64 x 16
  static constexpr int A_BOX_MAX = 64 * 4 * 128;    // ws = 64: 4 rows of 64 pixels (ws = 32: 6 x 32;
                                                    // the stem: 4 rows of 128 pixels x 32 bytes)
  static constexpr int A_STAGE = A_BOX_MAX + 1024;  // + the last tap window's over-read (the stem)
  static constexpr int STAGES = 3;
  static constexpr int STAGING_BYTES = kEpiWarps * 4096;  // one 32 x 64 tile per epilogue warp
  // 3x3: rows 0 and 1 of each warp's shifted partials (128 32-bit columns),
  // per epilogue group, tile parity and TMEM sub-partition
  static constexpr int XCH_BYTES = 2 * 2 * 4 * 2 * 512;
  static constexpr int BAR_BYTES = 8 * (2 * STAGES + 7) + 16;
  static constexpr int SMEM = 1024 + B_BYTES + STAGES * A_STAGE + STAGING_BYTES + XCH_BYTES + BAR_BYTES;
  static_assert(SMEM <= 232448, "shared memory per CTA");
};

// 3x3 halo epilogue.  The accumulator holds in columns 64 j + c (j = 0, 1, 2)
// the products of taps (r, j) read through the window of tap (r, 0), summed
// over the filter rows r: row m of it is tap column j's share of output row
// m - j.  So output m = D[m][c] + D[m + 1][64 + c] + D[m + 2][128 + c], each
// addition rounded to FP16 (an FP32 accumulator: added in FP32 and rounded
// once).  Rows m + 1 and m + 2 come from lanes + 1 and + 2 of the warp, and
// for lanes 30 and 31 from rows 0 and 1 of the next warp (nxt: its rows
// continue the same padded row), which that warp left in shared memory at
// `other` (row l at + l * 512 bytes, columns 64..191 as 32-bit words).  Rows
// m + 1, m + 2 of a padded row's last real pixels are still in that padded
// row (ws >= W + 2), so a tile never needs another tile's rows.
__device__ __forceinline__ void halo3_publish(uint32_t tb, int lane, uint32_t mine) {
#pragma unroll 1
  for (int h = 0; h < 2; ++h) {
    uint32_t v[64];
    tmem_ld16(tb + 64 + 64 * h, v);
    tmem_ld16(tb + 80 + 64 * h, v + 16);
    tmem_ld16(tb + 96 + 64 * h, v + 32);
    tmem_ld16(tb + 112 + 64 * h, v + 48);
    tmem_ld_wait();
    if (lane < 2) {
#pragma unroll
      for (int q = 0; q < 16; ++q)
        st_shared_v4(mine + (uint32_t)(lane * 512 + (64 * h + 4 * q) * 4),
                     make_uint4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]));
    }
  }
}

__device__ __forceinline__ void halo3_combine(uint32_t tb, int lane, bool f32, bool nxt, uint32_t other,
                                              uint32_t* o) {
#pragma unroll
  for (int c = 0; c < 64; c += 16) {
    uint32_t d0[16], a[16], b[16];
    tmem_ld16(tb + c, d0);
    tmem_ld16(tb + 64 + c, a);
    tmem_ld16(tb + 128 + c, b);
    tmem_ld_wait();
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      a[j] = __shfl_down_sync(0xffffffffu, a[j], 1);
      b[j] = __shfl_down_sync(0xffffffffu, b[j], 2);
    }
    if (nxt && lane >= 30) {
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        uint4 v;
        if (lane == 31) {
          ld_shared_v4(other + (uint32_t)((c + 4 * q) * 4), v);
          a[4 * q] = v.x, a[4 * q + 1] = v.y, a[4 * q + 2] = v.z, a[4 * q + 3] = v.w;
        }
        ld_shared_v4(other + (uint32_t)((lane - 30) * 512 + (64 + c + 4 * q) * 4), v);
        b[4 * q] = v.x, b[4 * q + 1] = v.y, b[4 * q + 2] = v.z, b[4 * q + 3] = v.w;
      }
    }
    if (f32) {
#pragma unroll
      for (int j = 0; j < 16; ++j)
        d0[j] = __float_as_uint(
            __fadd_rn(__fadd_rn(__uint_as_float(d0[j]), __uint_as_float(a[j])), __uint_as_float(b[j])));
      f32_to_f16_lo<16>(d0);
#pragma unroll
      for (int j = 0; j < 8; ++j) o[c / 2 + j] = pack_lo(d0[2 * j], d0[2 * j + 1]);
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j)
        o[c / 2 + j] = hadd2_rn(hadd2_rn(pack_lo(d0[2 * j], d0[2 * j + 1]), pack_lo(a[2 * j], a[2 * j + 1])),
                                pack_lo(b[2 * j], b[2 * j + 1]));
    }
  }
}

// CB = bytes of one input pixel: 128 (3x3, nine taps of four K = 16 steps,
// 128-byte swizzle) or 32 (the space-to-depth stem, sixteen taps of one step,
// 32-byte swizzle).  The MMA issue loop is unrolled over taps and steps with
// descriptors formed by adding 16-byte offsets to two base descriptors (the
// start-address field is the low 14 bits; desc_addr16 masks a shared address
// into it, and a stage plus its tap offsets stays below 256 KB), so a single
// thread keeps up with N = 64 MMAs.
template <int CB, bool BS>
__global__ void __launch_bounds__(kGemmThreads, 1)
    k_gemm_halo(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB,
                const __grid_constant__ CUtensorMap mapC, const __grid_constant__ GemmParams p) {
  using Cfg = HaloCfg;
  constexpr int NTAPS = CB == 128 ? 9 : 16;
  constexpr int KSTEPS = CB / 32;                 // K = 16 steps per tap
  constexpr uint32_t SWZ = CB == 128 ? 2u : 6u;   // descriptor swizzle code
  constexpr int B_TILE = 64 * CB;                 // one tap's 64-row weight slice
  constexpr int ACC = CB == 128 ? 192 : 64;       // accumulator columns (3x3: three taps' slices)
  constexpr int TMEM_COLS = CB == 128 ? 512 : 128;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* bres = smem;                                   // the taps' weight slices
  uint8_t* astages = smem + Cfg::B_BYTES;                 // 1024-aligned stages
  uint8_t* staging = astages + Cfg::STAGES * Cfg::A_STAGE;
  uint8_t* xch = staging + Cfg::STAGING_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(xch + Cfg::XCH_BYTES);
  uint64_t* full = bars;
  uint64_t* empty = bars + Cfg::STAGES;
  uint64_t* tfull = bars + 2 * Cfg::STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* bready = tempty + 2;
  uint64_t* xbar = bready + 1;  // per epilogue group: the exchange of shifted partials
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(xbar + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int ws = p.halo_ws, rows = kBM / ws;
  const uint32_t box_bytes = (uint32_t)(p.halo_box_rows * ws * CB);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < Cfg::STAGES; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&tfull[a]), 1);
      mbar_init(smem_u32(&tempty[a]), 4);
      mbar_init(smem_u32(&xbar[a]), 4);
    }
    mbar_init(smem_u32(bready), 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&mapA);
    tma_prefetch_desc(&mapB);
    tma_prefetch_desc(&mapC);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), TMEM_COLS);
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
      // resident weights: the 64-row slice of each tap
      const uint32_t bb = smem_u32(bready);
      mbar_arrive_expect_tx(bb, (uint32_t)(NTAPS * B_TILE));
      for (int t = 0; t < NTAPS; ++t) {
        const uint32_t dst = smem_u32(bres + t * B_TILE);
        if (p.b_mode == LD_TILED_K)
          tma_load_2d(dst, &mapB, bb, p.tap_w[t] * (CB / 2), 0);
        else
          tma_load_3d(dst, &mapB, bb, 0, p.tap_w[t], 0);
      }
      int stage = 0;
      uint32_t phase = 0, issued = 0;
      for (int u = blockIdx.x; u < total && !*abort_flag; u += gridDim.x) {
        const int g = u * rows;  // first image row of the tile over all images (n*H + i0)
        const int n = g / p.halo_h, i0 = g - n * p.halo_h;
        if (!mbar_wait(smem_u32(&empty[stage]), phase ^ 1, lim)) {
          record_timeout(p, abort_flag);
          break;
        }
        const uint32_t fb = smem_u32(&full[stage]);
        mbar_arrive_expect_tx(fb, box_bytes);
        tma_load_4d(smem_u32(astages + stage * Cfg::A_STAGE), &mapA, fb, 0, p.halo_col0, i0 + p.halo_row0, n);
        ++issued;
        if (++stage == Cfg::STAGES) {
          stage = 0;
          phase ^= 1;
        }
      }
      // let every copy this thread started land before the CTA can exit
      mbar_wait(smem_u32(bready), 0, 1000000000ull);
      if (*abort_flag) {
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
      bool ok = mbar_wait(smem_u32(bready), 0, lim);
      if (!ok) record_timeout(p, abort_flag);
      tc_fence_after();
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      // tap windows in 16-byte units, and the two base descriptors
      uint32_t toff[NTAPS];
#pragma unroll
      for (int t = 0; t < NTAPS; ++t) toff[t] = (uint32_t)((p.tap_dr[t] * ws + p.tap_ds[t]) * CB) >> 4;
      const uint64_t adesc0 = smem_desc(0, 16, 8 * CB, SWZ);
      const uint64_t bdesc0 = smem_desc(smem_u32(bres), p.b_lbo, p.b_sbo, SWZ);
      const uint32_t bk16 = (uint32_t)p.b_kstep >> 4;
      for (int u = blockIdx.x; ok && u < total && !*abort_flag; u += gridDim.x) {
        if (!mbar_wait(smem_u32(&tempty[acc]), acc_phase ^ 1, lim) ||
            !mbar_wait(smem_u32(&full[stage]), phase, lim)) {
          record_timeout(p, abort_flag);
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * ACC);
        const uint64_t abase = adesc0 + desc_addr16(smem_u32(astages + stage * Cfg::A_STAGE));
        if constexpr (CB == 128) {
          // filter row r: one N = 192 MMA per K step, the window of tap (r, 0)
          // against the contiguous slices of taps (r, 0), (r, 1), (r, 2)
#pragma unroll
          for (int r = 0; r < 3; ++r)
#pragma unroll
            for (int kk = 0; kk < KSTEPS; ++kk)
              tc_mma_f16(d_tmem, abase + toff[3 * r] + kk * 2,
                         bdesc0 + (uint32_t)(3 * r * (B_TILE >> 4)) + kk * bk16, p.idesc,
                         (r > 0 || kk > 0) ? 1u : 0u);
        } else {
#pragma unroll
          for (int t = 0; t < NTAPS; ++t)
#pragma unroll
            for (int kk = 0; kk < KSTEPS; ++kk)
              tc_mma_f16(d_tmem, abase + toff[t] + kk * 2, bdesc0 + (uint32_t)(t * (B_TILE >> 4)) + kk * bk16,
                         p.idesc, (t > 0 || kk > 0) ? 1u : 0u);
        }
        tc_commit(smem_u32(&empty[stage]));
        if (++stage == Cfg::STAGES) {
          stage = 0;
          phase ^= 1;
        }
        tc_commit(smem_u32(&tfull[acc]));
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1;
      }
    }
  } else {
    // epilogue warps 2..9: group (w - 2) / 4 drains accumulator 0 or 1 (the
    // CTA's even or odd tiles), warp w its TMEM sub-partition w % 4; 32 rows
    // each, which lie in one image row of the padded grid (ws is a multiple of 32)
    const int e = warp - 2, grp = e >> 2, sub = warp & 3;
    const int acc = grp;
    uint32_t acc_phase = 0;
    const uint32_t stg = smem_u32(staging) + (uint32_t)(e * 4096);
    EpiStats stats;
    stats.init();
    BwdIn bin;
    // 3x3: exchange of shifted partials between the warps of a padded row
    // (none at ws = 32, where a warp holds a whole padded row); xit counts
    // this warp's tiles (exchange buffer and barrier parity)
    const bool xchg = CB == 128 && ws > 32;
    const bool pub = xchg && (sub * 32) % ws != 0;
    const bool nxt = xchg && (sub * 32 + 32) % ws != 0;
    uint32_t xit = 0;
    for (int u = blockIdx.x + grp * gridDim.x; u < total; u += 2 * gridDim.x) {
      if (__any_sync(0xffffffffu, *abort_flag != 0)) break;
      if (BS && p.st_mean) {  // the tile's inputs, loaded while the accumulator is computed
        const int mp = u * kBM + sub * 32;
        const int nv0 = min(32, max(0, p.halo_w - mp % ws));
        // pixel of padded row mp: image row mp / ws, column mp % ws
        if (nv0 > 0) bin.load(p, (long long)(mp / ws) * p.halo_w + mp % ws, 0, nv0, lane);
      }
      const bool got = mbar_wait(smem_u32(&tfull[acc]), acc_phase, lim);
      if (!__all_sync(0xffffffffu, got)) {
        if (lane == 0) record_timeout(p, abort_flag);
        break;
      }
      tc_fence_after();
      const uint32_t tbase = tmem_base + ((uint32_t)(sub * 32) << 16) + (uint32_t)(acc * ACC);
      uint32_t o[32];  // the warp's 32 rows x 64 outputs, FP16 pairs
      if constexpr (CB == 128) {
        const uint32_t xslot = smem_u32(xch) + (uint32_t)((grp * 2 + (int)(xit & 1)) * 4 * 1024);
        if (xchg) {
          if (pub) halo3_publish(tbase, lane, xslot + (uint32_t)(sub * 1024));
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&xbar[grp]));
          const bool okx = mbar_wait(smem_u32(&xbar[grp]), xit & 1, lim);
          if (!__all_sync(0xffffffffu, okx)) {
            if (lane == 0) record_timeout(p, abort_flag);
            break;
          }
        }
        halo3_combine(tbase, lane, p.d_f32 != 0, nxt, xslot + (uint32_t)((sub + 1) * 1024), o);
        ++xit;
      } else {
        uint32_t r[64];
        tmem_ld16(tbase, r);
        tmem_ld16(tbase + 16, r + 16);
        tmem_ld16(tbase + 32, r + 32);
        tmem_ld16(tbase + 48, r + 48);
        tmem_ld_wait();
        if (p.d_f32) f32_to_f16_lo<64>(r);  // FP32 accumulator: one rounding to FP16
#pragma unroll
        for (int j = 0; j < 32; ++j) o[j] = pack_lo(r[2 * j], r[2 * j + 1]);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&tempty[acc]));
      if (lane == 0) bulk_wait_read0();  // the previous store has read the staging tile
      __syncwarp();
#pragma unroll
      for (int j = 0; j < 8; ++j)
        st_shared_v4(stg + lane * 128 + ((j ^ (lane & 7)) << 4),
                     make_uint4(o[j * 4], o[j * 4 + 1], o[j * 4 + 2], o[j * 4 + 3]));
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        const int mp = u * kBM + sub * 32;  // first padded-grid row of the warp
        const int grow = mp / ws, col = mp - grow * ws;
        if (col < p.halo_w) {  // a box wholly right of the image has nothing to store
          tma_store_3d(&mapC, stg, 0, col, grow);
          bulk_commit();
        }
      }
      if (p.st_mean) {
        const int mp = u * kBM + sub * 32;
        const int nv = min(32, max(0, p.halo_w - mp % ws));  // columns j >= W are padding
        if (nv > 0) {
          if (BS)
            stats.leaf_bwd(0, stg, lane, nv, bin);
          else
            stats.leaf(0, stg, lane, nv);
          stats.end_tile(nv);
        }
      }
      acc_phase ^= 1;
    }
    if (lane == 0) bulk_wait0();
    if (p.st_mean) {
      if (BS)
        stats.write_cta_bwd(p, staging, e, blockIdx.x, 0, 1, lane, p.bs_levels);
      else
        stats.write_cta(p, staging, e, blockIdx.x, 0, 1, lane, true);
      if (blockIdx.x == 0 && e == 0 && lane == 0) {
        p.st_hdr[0] = (int)gridDim.x;
        p.st_hdr[1] = 5 + p.bs_levels + 3;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

cudaError_t launch_gemm_halo(const CUtensorMap& mA, const CUtensorMap& mB, const CUtensorMap& mC,
                             const GemmParams& p, int grid, cudaStream_t s) {
  // the resident weights, the A box and its furthest tap window must fit their buffers
  const int max_off = [&] {
    int m = 0;
    for (int t = 0; t < p.ntaps; ++t) m = max(m, (p.tap_dr[t] * p.halo_ws + p.tap_ds[t]) * p.halo_cb);
    return m;
  }();
  if (p.ntaps != (p.halo_cb == 128 ? 9 : 16) || (p.halo_cb != 128 && p.halo_cb != 32) || p.halo_ws <= 0 ||
      kBM % p.halo_ws != 0 || p.ntaps * 64 * p.halo_cb > HaloCfg::B_BYTES ||
      p.halo_box_rows * p.halo_ws * p.halo_cb > HaloCfg::A_BOX_MAX ||
      max_off + kBM * p.halo_cb > HaloCfg::A_STAGE)
    return cudaErrorInvalidValue;
  // 3x3: slot t holds tap (t / 3, t % 3), so filter row r's three slices are
  // the contiguous N = 192 operand read through tap (r, 0)'s window
  if (p.halo_cb == 128)
    for (int t = 0; t < 9; ++t)
      if (p.tap_dr[t] != t / 3 || p.tap_ds[t] != t % 3) return cudaErrorInvalidValue;
  // variants: 128-byte pixels, with backward statistics (the 3x3 data gradient) or not; 32-byte pixels
  static bool attr_set[3][64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  const int v = p.halo_cb == 128 ? (p.bs_x ? 1 : 0) : 2;
  if (v == 2 && p.bs_x) return cudaErrorInvalidValue;
  void (*const kern[3])(CUtensorMap, CUtensorMap, CUtensorMap, GemmParams) = {
      k_gemm_halo<128, false>, k_gemm_halo<128, true>, k_gemm_halo<32, false>};
  if (dev < 64 && !attr_set[v][dev]) {
    cudaError_t e = cudaFuncSetAttribute(kern[v], cudaFuncAttributeMaxDynamicSharedMemorySize, HaloCfg::SMEM);
    if (e != cudaSuccess) return e;
    attr_set[v][dev] = true;
  }
  launch_pdl(kern[v], dim3(grid), dim3(kGemmThreads), HaloCfg::SMEM, s, mA, mB, mC, p);
  return counted_launches(1);
}

// ---------------------------------------------------------------------------
// Stem weight gradient on the space-to-depth input (the stem forward's xs:
// N x Hs x Ws x 16, Hs = P + 3).  With dy on a padded grid of ws = 128
// columns per output row (columns >= Q zero), tap (u, v) of the 4x4 form is
//   dW'[k][u][v][ch] = sum_p dy[p][k] * xs[p + u*ws + v][ch],
// p over the padded pixels of every output row.  One MMA (M = 128, N = 64,
// K = 16 pixels, both operands MN-major) yields two tap rows at once:
//   A = the 64 channels of dy at pixels p - ws (M rows 0..63) and p (rows
//       64..127): two 128-byte-swizzled M atoms one padded row apart (LBO);
//   B = xs at p + u*ws + v for v = 0..3: four 16-channel N atoms one pixel
//       (32 bytes, LBO) apart, 32-byte swizzle.
// Rows 64..127 then accumulate tap (u, v) over output row i, rows 0..63 tap
// (u + 1, v) over output row i - 1; u = 0 and u = 2 cover all sixteen taps
// when i runs over 0..P (dy rows -1 and P read as zeros).  A work unit is
// one (image, i) row: a stage holds dy rows i - 1, i (2 x 128 x 128 B) and
// xs rows i .. i + 3 (4 x 128 x 32 B; windows reach at most 3 pixels into
// row i + 3, and only at padding columns, where dy is zero).  Units are
// accumulated in FP16 in TMEM over chunks of p.kb_per_split rows (4,096
// padded pixels at ws = 128), and each chunk's 128 x 128 FP16 partial
// [(a, k)][(u/2, v, ch)] goes to p.out + chunk * 128 * 128 for the split-K
// tree.  Same roles and bounded waits as k_gemm_halo.
// ---------------------------------------------------------------------------
struct StemWgradCfg {
  static constexpr int WS = 128;
  static constexpr int DY_BYTES = 2 * WS * 128;   // dy rows i - 1, i
  static constexpr int XS_BYTES = 4 * WS * 32;    // xs rows i .. i + 3
  static constexpr int STAGE = DY_BYTES + XS_BYTES;
  static constexpr int STAGES = 4;
  static constexpr int TMEM_COLS = 256;           // two 128-column accumulators
  static constexpr int BAR_BYTES = 8 * (2 * STAGES + 4) + 16;
  static constexpr int SMEM = 1024 + STAGES * STAGE + BAR_BYTES;
};
constexpr int kStemWgradThreads = 192;

__global__ void __launch_bounds__(kStemWgradThreads, 1)
    k_stem_wgrad(const __grid_constant__ CUtensorMap mapDy, const __grid_constant__ CUtensorMap mapXs,
                 const __grid_constant__ GemmParams p) {
  using Cfg = StemWgradCfg;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Cfg::STAGES * Cfg::STAGE);
  uint64_t* full = bars;
  uint64_t* empty = bars + Cfg::STAGES;
  uint64_t* tfull = bars + 2 * Cfg::STAGES;
  uint64_t* tempty = tfull + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
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
    tma_prefetch_desc(&mapXs);
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
  const int rows_total = p.num_kb;      // (P + 1) * N row units
  const int per_chunk = p.kb_per_split; // row units per accumulator
  const int chunks = p.m_tiles;
  const int rows_img = p.halo_h + 1;    // i = 0 .. P
  const uint64_t lim = p.wait_limit_ns;

  if (warp == 0) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0, issued = 0;
      for (int c = blockIdx.x; c < chunks && !*abort_flag; c += gridDim.x) {
        const int g1 = min(rows_total, (c + 1) * per_chunk);
        for (int g = c * per_chunk; g < g1 && !*abort_flag; ++g) {
          const int n = g / rows_img, i = g - n * rows_img;
          if (!mbar_wait(smem_u32(&empty[stage]), phase ^ 1, lim)) {
            record_timeout(p, abort_flag);
            break;
          }
          const uint32_t fb = smem_u32(&full[stage]);
          const uint32_t dst = smem_u32(smem + stage * Cfg::STAGE);
          mbar_arrive_expect_tx(fb, (uint32_t)Cfg::STAGE);
          tma_load_4d(dst, &mapDy, fb, 0, 0, i - 1, n);
          tma_load_4d(dst + Cfg::DY_BYTES, &mapXs, fb, 0, 0, i, n);
          ++issued;
          if (++stage == Cfg::STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (*abort_flag) {  // let every copy this thread started land before the CTA can exit
        const uint32_t nn = issued < (uint32_t)Cfg::STAGES ? issued : (uint32_t)Cfg::STAGES;
        int s = stage;
        uint32_t ph = phase;
        for (uint32_t q = 0; q < nn; ++q) {
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
      // A: dy, MN-major 128-byte swizzle, M atoms one padded row (ws * 128 B)
      // apart, 8-pixel K groups 1 KB apart; B: xs, MN-major 32-byte swizzle,
      // N atoms one pixel (32 B) apart, 8-pixel K groups 256 B apart
      const uint64_t adesc0 = smem_desc(0, Cfg::WS * 128, 1024, 2);
      const uint64_t bdesc0 = smem_desc(0, 32, 256, 6);
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int c = blockIdx.x; ok && c < chunks && !*abort_flag; c += gridDim.x) {
        if (!mbar_wait(smem_u32(&tempty[acc]), acc_phase ^ 1, lim)) {
          record_timeout(p, abort_flag);
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * 128);
        const int g0 = c * per_chunk, g1 = min(rows_total, (c + 1) * per_chunk);
        for (int g = g0; g < g1; ++g) {
          if (!mbar_wait(smem_u32(&full[stage]), phase, lim)) {
            record_timeout(p, abort_flag);
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa16 = desc_addr16(smem_u32(smem + stage * Cfg::STAGE));
          const uint64_t ab = adesc0 + sa16;
          const uint64_t bb = bdesc0 + sa16 + (Cfg::DY_BYTES >> 4);
#pragma unroll
          for (int js = 0; js < Cfg::WS / 16; ++js)
#pragma unroll
            for (int uu = 0; uu < 2; ++uu)
              tc_mma_f16(d_tmem + (uint32_t)(uu * 64), ab + (uint32_t)(js * (2048 >> 4)),
                         bb + (uint32_t)((uu * 2 * Cfg::WS * 32 + js * 512) >> 4), p.idesc,
                         (g > g0 || js > 0) ? 1u : 0u);
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
    }
  } else {
    // epilogue warps 2..5 -> TMEM sub-partitions 2, 3, 0, 1: row = (a, k)
    const int sub = warp & 3;
    const int row = sub * 32 + lane;
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int c = blockIdx.x; c < chunks; c += gridDim.x) {
      if (__any_sync(0xffffffffu, *abort_flag != 0)) break;
      const bool got = mbar_wait(smem_u32(&tfull[acc]), acc_phase, lim);
      if (!__all_sync(0xffffffffu, got)) {
        if (lane == 0) record_timeout(p, abort_flag);
        break;
      }
      tc_fence_after();
      uint4* dst = reinterpret_cast<uint4*>(p.out + ((size_t)c * 128 + row) * 128);
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        const uint32_t tbase = tmem_base + ((uint32_t)(sub * 32) << 16) + (uint32_t)(acc * 128 + half * 64);
        uint32_t r[64];
        tmem_ld16(tbase, r);
        tmem_ld16(tbase + 16, r + 16);
        tmem_ld16(tbase + 32, r + 32);
        tmem_ld16(tbase + 48, r + 48);
        tmem_ld_wait();
        if (p.d_f32) f32_to_f16_lo<64>(r);  // FP32 accumulator: one rounding to FP16
#pragma unroll
        for (int j = 0; j < 8; ++j)
          dst[half * 8 + j] = make_uint4(pack_lo(r[j * 8 + 0], r[j * 8 + 1]), pack_lo(r[j * 8 + 2], r[j * 8 + 3]),
                                         pack_lo(r[j * 8 + 4], r[j * 8 + 5]), pack_lo(r[j * 8 + 6], r[j * 8 + 7]));
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&tempty[acc]));
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

cudaError_t launch_stem_wgrad(const CUtensorMap& mDy, const CUtensorMap& mXs, const GemmParams& p, int grid,
                              cudaStream_t s) {
  if (p.halo_ws != StemWgradCfg::WS || p.kb_per_split < 1 || p.m_tiles < 1 || grid < 1) return cudaErrorInvalidValue;
  static bool attr_set[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 64 && !attr_set[dev]) {
    cudaError_t e = cudaFuncSetAttribute(k_stem_wgrad, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         StemWgradCfg::SMEM);
    if (e != cudaSuccess) return e;
    attr_set[dev] = true;
  }
  launch_pdl(k_stem_wgrad, dim3(grid), dim3(kStemWgradThreads), StemWgradCfg::SMEM, s, mDy, mXs, p);
  return counted_launches(1);
}

// ---------------------------------------------------------------------------
// Weight gradient of the 3x3 / stride 1 / pad 1 convolution with 64 input and
// 64 output channels (the 56x56 layers of ResNet-50), on padded rows of
// ws = 64 pixels (W + 2 <= ws).  Output pixel (i, j) is padded pixel p = i*ws + j
// of dy (zero at j >= W); the input grid holds x[i][j' - 1] at column j'
// (zero outside the image), so that
//   dW[k][r][s][c] = sum_p dy[p][k] * xp[p + (r - 1)*ws + s][c].
// One MMA (M = 128, N = 192, K = 16 pixels, both operands MN-major, 128-byte
// swizzle) covers three filter columns and two filter rows:
//   A = the 64 channels of dy at pixels p - ws (M rows 0..63) and p (rows
//       64..127): two M atoms one padded row apart (LBO = ws * 128 B);
//   B = the input at p + u*ws + s - ws for s = 0, 1, 2: three 64-channel N
//       atoms one pixel apart (LBO = 128 B; the 128-byte swizzle is a function
//       of the absolute address, so a window may start at any row).
// For output row i, u = 0 accumulates filter row 0 in M rows 64..127 (dy row i
// against input row i - 1) and filter row 1 in rows 0..63 (dy row i - 1 against
// input row i - 1); u = 1 accumulates filter row 2 in rows 0..63 (the same
// product for rows 64..127, filter row 1 again, is discarded).  Summing over
// i = 0 .. P (dy rows -1 and P read as zeros) covers every term once.  A unit
// is two output rows (i0, i0 + 1) of one image: a stage holds dy rows
// i0 - 1 .. i0 + 1 (3 x 64 x 128 B) and input rows i0 - 1 .. i0 + 2
// (4 x 64 x 128 B; a window reaches past its row only at columns where dy is
// zero).  Units are accumulated in FP16 in TMEM (two 192-column accumulators,
// u = 0 and 1) over chunks of p.kb_per_split units (4,096 padded pixels), and
// each chunk's 64 x 576 partial [k][(r, s, c)] goes to p.out + chunk * 64 * 576
// for the split-K tree, laid out as the weight gradient itself.  Roles and
// bounded waits as k_stem_wgrad; the accumulators are single-buffered (2 x 192
// of the 512 columns), so a chunk's MMAs wait for the previous chunk's drain.
// ---------------------------------------------------------------------------
struct Wgrad3Cfg {
  static constexpr int WS = 64;
  static constexpr int DY_BYTES = 3 * WS * 128;  // dy rows i0 - 1 .. i0 + 1
  static constexpr int X_BYTES = 4 * WS * 128;   // input rows i0 - 1 .. i0 + 2
  static constexpr int STAGE = DY_BYTES + X_BYTES;
  static constexpr int STAGES = 4;
  static constexpr int TMEM_COLS = 512;          // accumulators u = 0, 1 at columns 0 and 192
  static constexpr int BAR_BYTES = 8 * (2 * STAGES + 2) + 16;
  static constexpr int SMEM = 1024 + STAGES * STAGE + BAR_BYTES;
  static_assert(SMEM <= 232448, "shared memory per CTA");
};
constexpr int kWgrad3Threads = 192;

__global__ void __launch_bounds__(kWgrad3Threads, 1)
    k_wgrad3x3_halo(const __grid_constant__ CUtensorMap mapDy, const __grid_constant__ CUtensorMap mapX,
                    const __grid_constant__ GemmParams p) {
  using Cfg = Wgrad3Cfg;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Cfg::STAGES * Cfg::STAGE);
  uint64_t* full = bars;
  uint64_t* empty = bars + Cfg::STAGES;
  uint64_t* tfull = bars + 2 * Cfg::STAGES;
  uint64_t* tempty = tfull + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < Cfg::STAGES; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    mbar_init(smem_u32(tfull), 1);
    mbar_init(smem_u32(tempty), 4);
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
  const int units = p.num_kb;            // N * ceil((P + 1) / 2) two-row units
  const int per_chunk = p.kb_per_split;  // units per accumulation
  const int chunks = p.m_tiles;
  const int upi = (p.halo_h + 2) / 2;    // units per image: output rows i = 0 .. P in pairs
  const uint64_t lim = p.wait_limit_ns;

  if (warp == 0) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0, issued = 0;
      for (int c = blockIdx.x; c < chunks && !*abort_flag; c += gridDim.x) {
        const int g1 = min(units, (c + 1) * per_chunk);
        for (int g = c * per_chunk; g < g1 && !*abort_flag; ++g) {
          const int n = g / upi, i0 = 2 * (g - n * upi);
          if (!mbar_wait(smem_u32(&empty[stage]), phase ^ 1, lim)) {
            record_timeout(p, abort_flag);
            break;
          }
          const uint32_t fb = smem_u32(&full[stage]);
          const uint32_t dst = smem_u32(smem + stage * Cfg::STAGE);
          mbar_arrive_expect_tx(fb, (uint32_t)Cfg::STAGE);
          tma_load_4d(dst, &mapDy, fb, 0, 0, i0 - 1, n);
          tma_load_4d(dst + Cfg::DY_BYTES, &mapX, fb, 0, -1, i0 - 1, n);
          ++issued;
          if (++stage == Cfg::STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (*abort_flag) {  // let every copy this thread started land before the CTA can exit
        const uint32_t nn = issued < (uint32_t)Cfg::STAGES ? issued : (uint32_t)Cfg::STAGES;
        int s = stage;
        uint32_t ph = phase;
        for (uint32_t q = 0; q < nn; ++q) {
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
      // A: dy, MN-major 128-byte swizzle, M atoms one padded row apart, 8-pixel
      // K groups 1 KB apart; B: the input, three N atoms one pixel apart
      const uint64_t adesc0 = smem_desc(0, Cfg::WS * 128, 1024, 2);
      const uint64_t bdesc0 = smem_desc(0, 128, 1024, 2);
      int stage = 0;
      uint32_t phase = 0, acc_phase = 0;
      bool ok = true;
      for (int c = blockIdx.x; ok && c < chunks && !*abort_flag; c += gridDim.x) {
        if (!mbar_wait(smem_u32(tempty), acc_phase ^ 1, lim)) {
          record_timeout(p, abort_flag);
          break;
        }
        tc_fence_after();
        const int g0 = c * per_chunk, g1 = min(units, (c + 1) * per_chunk);
        for (int g = g0; g < g1; ++g) {
          if (!mbar_wait(smem_u32(&full[stage]), phase, lim)) {
            record_timeout(p, abort_flag);
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa16 = desc_addr16(smem_u32(smem + stage * Cfg::STAGE));
          const uint64_t ab = adesc0 + sa16;
          const uint64_t bb = bdesc0 + sa16 + (Cfg::DY_BYTES >> 4);
#pragma unroll
          for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int js = 0; js < Cfg::WS / 16; ++js)
#pragma unroll
              for (int u = 0; u < 2; ++u)
                tc_mma_f16(tmem_base + (uint32_t)(u * 192), ab + (uint32_t)((h * Cfg::WS * 128 + js * 2048) >> 4),
                           bb + (uint32_t)(((h + u) * Cfg::WS * 128 + js * 2048) >> 4), p.idesc,
                           (g > g0 || h > 0 || js > 0) ? 1u : 0u);
          tc_commit(smem_u32(&empty[stage]));
          if (++stage == Cfg::STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        tc_commit(smem_u32(tfull));
        acc_phase ^= 1;
      }
    }
  } else {
    // epilogue warps 2..5 -> TMEM sub-partitions 2, 3, 0, 1.  Row m < 64: k = m,
    // filter rows 1 (u = 0) and 2 (u = 1); m >= 64: k = m - 64, filter row 0 (u = 0).
    const int sub = warp & 3;
    const int m = sub * 32 + lane;
    const int k = m & 63;
    uint32_t acc_phase = 0;
    for (int c = blockIdx.x; c < chunks; c += gridDim.x) {
      if (__any_sync(0xffffffffu, *abort_flag != 0)) break;
      const bool got = mbar_wait(smem_u32(tfull), acc_phase, lim);
      if (!__all_sync(0xffffffffu, got)) {
        if (lane == 0) record_timeout(p, abort_flag);
        break;
      }
      tc_fence_after();
      uint16_t* prow = p.out + ((size_t)c * 64 + k) * 576;
#pragma unroll 1
      for (int u = 0; u < 2; ++u) {
        if (u == 1 && m >= 64) continue;  // warp-uniform: sub-partitions 2, 3 hold rows 64..127
        const int r = u == 0 ? (m < 64 ? 1 : 0) : 2;
        uint4* dst = reinterpret_cast<uint4*>(prow + r * 192);
#pragma unroll 1
        for (int cc = 0; cc < 192; cc += 64) {
          const uint32_t tb = tmem_base + ((uint32_t)(sub * 32) << 16) + (uint32_t)(u * 192 + cc);
          uint32_t v[64];
          tmem_ld16(tb, v);
          tmem_ld16(tb + 16, v + 16);
          tmem_ld16(tb + 32, v + 32);
          tmem_ld16(tb + 48, v + 48);
          tmem_ld_wait();
          if (p.d_f32) f32_to_f16_lo<64>(v);  // FP32 accumulator: one rounding to FP16
#pragma unroll
          for (int j = 0; j < 8; ++j)
            dst[cc / 8 + j] = make_uint4(pack_lo(v[j * 8 + 0], v[j * 8 + 1]), pack_lo(v[j * 8 + 2], v[j * 8 + 3]),
                                         pack_lo(v[j * 8 + 4], v[j * 8 + 5]), pack_lo(v[j * 8 + 6], v[j * 8 + 7]));
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(tempty));
      acc_phase ^= 1;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, Cfg::TMEM_COLS);
  }
}

cudaError_t launch_wgrad3x3_halo(const CUtensorMap& mDy, const CUtensorMap& mX, const GemmParams& p, int grid,
                                 cudaStream_t s) {
  if (p.kb_per_split < 1 || p.m_tiles < 1 || grid < 1 || p.halo_h < 1) return cudaErrorInvalidValue;
  static bool attr_set[64] = {false};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 64 && !attr_set[dev]) {
    cudaError_t e = cudaFuncSetAttribute(k_wgrad3x3_halo, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         Wgrad3Cfg::SMEM);
    if (e != cudaSuccess) return e;
    attr_set[dev] = true;
  }
  launch_pdl(k_wgrad3x3_halo, dim3(grid), dim3(kWgrad3Threads), Wgrad3Cfg::SMEM, s, mDy, mX, p);
  return counted_launches(1);
}

}  // namespace pf16
