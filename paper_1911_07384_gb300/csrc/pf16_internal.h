// Internal interfaces of libpf16 shared between the C-ABI layer (pf16_api.cu)
// and the kernels (pf16_gemm.cu, pf16_elementwise.cu).  Not installed.
#pragma once
#include <atomic>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

namespace pf16 {

// Kernels this library has enqueued in the process (launches recorded into a
// CUDA graph during stream capture included).  Read by pf16_kernel_launches.
inline std::atomic<unsigned long long> g_kernel_launches{0};

// Launch with programmatic stream serialisation: the kernel may begin while
// the previous kernel of the stream drains; every kernel of the library calls
// pdl_wait() before it touches memory a predecessor writes.
template <typename... K, typename... A>
inline cudaError_t launch_pdl(void (*kernel)(K...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                              A&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<A&&>(args)...);
}

// Status of the n launches just made; they are counted when they succeeded.
inline cudaError_t counted_launches(int n) {
  const cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) g_kernel_launches.fetch_add((unsigned long long)n, std::memory_order_relaxed);
  return e;
}

// ---------------------------------------------------------------------------
// tcgen05 implicit-GEMM engine.
//
// D[m][n] = sum_k A[m][k] * B[n][k], D in FP16, accumulated in FP16 inside the
// tensor core (tcgen05.mma kind::f16, D type f16) into tensor memory.  Tiles
// are 128 (M) x BN (N) x 64 (K-block).  Each K-block of each operand is
// brought into shared memory by TMA in one of the load modes below, always as
// 128-byte-swizzled atoms of 8 rows x 128 bytes:
//   LD_TILED_K    2-D tiled box (64 k, rows): K-major operand, e.g. weights
//                 [K][R*S*C] or a dense [pixels][channels] activation.
//   LD_TILED_MN   2-D tiled boxes (64 mn, 64 k-rows): MN-major operand whose
//                 K-block is 64 consecutive rows, e.g. dy as [pixels][K].
//   LD_IM2COL_K   TMA im2col box (64 channels x 128 pixels) at one filter tap:
//                 K-major activation patch, the implicit-GEMM A of the
//                 forward and of the stride-phase data gradient.
//   LD_IM2COL_MN  TMA im2col boxes (64 channels x 64 pixels): MN-major
//                 activation patch for the weight gradient (K = pixels).
//   LD_TAP3D_MN   3-D tiled boxes over weights viewed as (C, R*S, K): the
//                 64(k) x 64(c) slice of one tap, MN-major B of the data
//                 gradient (no transposed weight copy is needed).
// ---------------------------------------------------------------------------
enum LoadMode : int {
  LD_TILED_K = 0,
  LD_TILED_MN = 1,
  LD_IM2COL_K = 2,
  LD_IM2COL_MN = 3,
  LD_TAP3D_MN = 4
};
enum OutMode : int { OUT_STORE = 0, OUT_ACCUM = 1, OUT_PARTIAL = 2 };

constexpr int kMaxTaps = 49;
constexpr int kBM = 128;
constexpr int kBK = 64;

// Pixel grid that GEMM rows (or K-block pixels) enumerate, image-major, and
// how a grid point maps to the im2col base coordinate (filter corner).
struct PixGrid {
  int gh, gw;             // grid points per image along h and w
  int step;               // input step between grid points (conv stride)
  int base_h, base_w;     // input coordinate of grid point (0, 0)
};

struct GemmParams {
  int M, N;               // GEMM output extent
  int num_kb;             // K-blocks in the whole reduction
  int kb_per_split;       // K-blocks per split (split-K)
  int splits;
  int m_tiles, n_tiles;
  int a_mode, b_mode;
  int a_cpt;              // IM2COL_K: channel chunks (of 64) per tap
  int b_cpt;              // TAP3D_MN: K chunks (of 64) per tap
  int b_cin;              // IM2COL_MN: input channels (n -> tap, channel)
  int b_oob_c;            // IM2COL_MN: a channel coordinate past the tensor (zero fill)
  PixGrid ga, gb;         // pixel grids of the im2col operands
  int ntaps;
  int8_t tap_dr[kMaxTaps], tap_ds[kMaxTaps];  // im2col offsets (h, w) of each tap
  int8_t tap_w[kMaxTaps];                     // weight tap index r*S+s (TAP3D_MN)
  // epilogue
  int out_mode;
  int tma_store;          // 1: rows written by TMA stores through mapC (row-major, no remap)
  uint16_t* out;
  long long ldo;          // output row stride (elements)
  int remap;              // rows -> strided positions of a stride phase
  int rm_gh, rm_gw, rm_H, rm_W, rm_step, rm_ph, rm_pw;
  // All stride phases of a data gradient in one launch (nphase > 1, with
  // remap and splits = nphase): a unit's split index is its phase f, whose
  // K-blocks are [ph_kb[f], ph_kb[f + 1]) of the phases' concatenated tap
  // lists and whose rows land at (i * rm_step + ph_h[f], j * rm_step + ph_w[f]).
  int nphase;
  int ph_kb[5];
  int8_t ph_h[4], ph_w[4];
  // MMA
  uint32_t idesc;
  int d_f32;              // FP32 accumulator in TMEM (PF16_F32_ACCUM), rounded once to FP16 in the epilogue
  uint32_t a_lbo, a_sbo, a_kstep;  // smem-descriptor strides, bytes per 16-wide k step
  uint32_t b_lbo, b_sbo, b_kstep;
  int* status;            // device status word
  unsigned long long wait_limit_ns;
  // halo mode (launch_gemm_halo): padded row width, output height and width,
  // bytes per pixel of the input (128: 64 channels, nine taps; 32: 16
  // channels, sixteen taps), rows of the A box, its start row / column
  // relative to the tile's first output row / column 0
  int halo_ws, halo_h, halo_w, halo_cb, halo_box_rows, halo_row0, halo_col0;
  // wide halo engine (launch_gemm_halo_wide): images side by side in one
  // padded row (1, or 4 for narrow images), padded columns per image, and
  // 64-channel chunks of the input
  int halo_ipr, halo_wi, halo_chunks;
  // BatchNorm forward statistics of the output (OUT_STORE through TMA only;
  // null when off): per epilogue warp a running (mean, variance, count) per
  // output channel over all its rows; the CTA's warps are merged at the end
  // and written as slot blockIdx / n_tiles; st_hdr[0] = number of slots.
  uint16_t* st_mean;      // [kBnStatSlots][N]
  uint16_t* st_var;       // [kBnStatSlots][N]
  int* st_cnt;            // [kBnStatSlots]
  int* st_hdr;
  // BatchNorm backward statistics instead (bs_x non-null; same buffer): the
  // output is the gradient dL/dy of a BatchNorm whose input bs_x ([pixels][N],
  // row pitch ldo), ReLU bits bs_mask ([pixels][N/8], or null) and saved
  // bs_mean / bs_invstd are given.  Per slot and channel: the pairwise sum
  // of dy' (in st_mean) and of dy' * xhat (in st_var), every epilogue warp's
  // tile trees padded with zeros to 2^bs_levels leaves; st_hdr[0] = slots,
  // st_hdr[1] = tree levels below the slot tree (5 + bs_levels + 3; informational).
  const uint16_t* bs_x;
  const uint8_t* bs_mask;
  const uint16_t* bs_mean;
  const uint16_t* bs_invstd;
  int bs_levels;
  // With the backward statistics only: an addend of the output, out =
  // rn(result + add_src) where add_mask's bit ([pixels][N/8], as bs_mask) is
  // set and out = rn(result + 0) elsewhere; add_src [pixels][N], pitch ldo.
  // The statistics are taken of that sum.  Null: no addend.
  const uint16_t* add_src;
  const uint8_t* add_mask;
  // BatchNorm applied in the operand path (xf_operand != 0; k_gemm's XF
  // variant): the operand's tiles hold a BatchNorm's input x, and before the
  // MMAs read a stage four transform warps replace each element of pixel row
  // r, channel c by the BatchNorm's output -- rn(rn(rn(gamma * rn(rn(x - mean)
  // * invstd)) + beta) * xf_scale), then ReLU when xf_relu -- the op sequence
  // of pf16_bn_fwd_bwd's apply, so the operand is bit-identical to the
  // BatchNorm's stored output.  Rows past xf_rows and channels past xf_C are
  // zero.  xf_operand 1: A (K-major, 128 pixel rows, the 64 channels of
  // K-block kb); 2: B (MN-major 64-pixel x 64-channel atoms of K-block kb,
  // channels n0 + 64 j).  With xf_mask (A only) the CTAs of n-tile 0 also
  // write the ReLU decisions in pf16_bn_fwd_bwd's bit-mask layout.
  int xf_operand;
  int xf_relu;
  uint16_t xf_scale;
  int xf_C;
  long long xf_rows;
  const uint16_t* xf_mean;
  const uint16_t* xf_invstd;
  const uint16_t* xf_gamma;
  const uint16_t* xf_beta;
  uint8_t* xf_mask;
};

// Conv-output BatchNorm statistics buffer (pf16_conv_fwd_bnstats): a header of
// 256 bytes (int slots), then mean and variance [kBnStatSlots][C] binary16 and
// counts [kBnStatSlots] int32, each section 256-byte aligned.
constexpr int kBnStatSlots = 256;
constexpr int kMaxTileTreeLevels = 12;  // an epilogue warp's tile trees hold fewer than 2^12 tiles
__host__ __device__ inline size_t bnstat_off_mean() { return 256; }
__host__ __device__ inline size_t bnstat_off_var(long long C) { return 256 + (size_t)kBnStatSlots * C * 2; }
__host__ __device__ inline size_t bnstat_off_cnt(long long C) {
  return 256 + (size_t)2 * kBnStatSlots * C * 2;
}
__host__ __device__ inline size_t bnstat_bytes(long long C) {
  return bnstat_off_cnt(C) + (size_t)kBnStatSlots * 4;
}

// Epilogue kinds of the conv GEMM (k_gemm's EPI).  The backward statistics
// take the TMA-fed epilogue for short reductions (at most kTmaEpiMaxKb
// K-blocks per tile: there the epilogue's traffic is the bound) and always
// with an addend; else their inputs go through registers, which leaves the
// main loop all of its pipeline stages.
enum GemmEpi : int { EPI_PLAIN = 0, EPI_BS = 1, EPI_BS_TMA = 2, EPI_BS_ADD = 3, EPI_BS_REMAP = 4 };
constexpr int kTmaEpiMaxKb = 8;
inline int gemm_epilogue(const GemmParams& p) {
  if (!p.bs_x) return EPI_PLAIN;
  if (p.add_src) return EPI_BS_ADD;
  if (p.remap) return EPI_BS_REMAP;  // scattered rows: x by cp.async into the same double buffers
  return p.kb_per_split <= kTmaEpiMaxKb ? EPI_BS_TMA : EPI_BS;
}

// The tensor-core rate probe (pf16_tc_rate): reps x 4 kind::f16 MMAs of
// M = 128, N = n per CTA, grid CTAs (one per SM).
cudaError_t launch_tc_rate(uint32_t idesc, int n, int chains, int reps, int grid, int* status,
                           unsigned long long wait_ns, cudaStream_t s);

// mapX / mapD: 128B-swizzled 32 x 64 boxes over bs_x and add_src ([M][N],
// pitch ldo), needed with the backward statistics (and the addend).
// Launch the engine (BN in {64, 128, 192, 256}) on `grid` persistent CTAs.
// Returns a cudaError_t.
cudaError_t launch_gemm(int BN, const CUtensorMap& mapA, const CUtensorMap& mapB,
                        const CUtensorMap& mapC, const GemmParams& p, int grid,
                        cudaStream_t stream, const CUtensorMap* mapX = nullptr,
                        const CUtensorMap* mapD = nullptr);
int gemm_smem_bytes(int BN);

// Halo engine for stride-1 convolutions with 64 outputs whose input pixel is
// 128 bytes (64 channels, 3x3 taps) or 32 bytes (16 channels, the stem after
// space-to-depth, 4x4 taps): A = one 4-D TMA box (channels x halo_ws columns
// x halo_box_rows rows) per 128-row tile of the padded pixel grid, taps as
// row-shifted descriptor windows, the taps' 64-row B slices resident; the
// output leaves through a 3-D map (64, Q, N*P) clipped at Q.  p.ntaps taps,
// p.tap_dr/tap_ds their window offsets, p.tap_w their weight tap; p.b_mode
// LD_TILED_K (weights [64][taps*C]) or LD_TAP3D_MN (weights (C, 9, K)).
// Stem weight gradient on the space-to-depth input: mapDy over dy (64, Q, P, N)
// with boxes (64, 128, 2, 1), mapXs over xs (16, Q + 3, P + 3, N) with boxes
// (16, 128, 4, 1); p.num_kb = N * (P + 1) row units, p.kb_per_split units per
// chunk, p.m_tiles chunks, p.halo_h = P, p.halo_ws = 128, p.out = the chunks'
// 128 x 128 FP16 partials.
// The 3x3 / stride 1 / pad 1, 64 -> 64 channel weight gradient on padded rows
// of 64 pixels (k_wgrad3x3_halo): p.num_kb two-row units, p.kb_per_split per
// chunk, p.m_tiles chunks, p.halo_h = P; partials [chunk][64][576] at p.out.
cudaError_t launch_wgrad3x3_halo(const CUtensorMap& mDy, const CUtensorMap& mX, const GemmParams& p, int grid,
                                 cudaStream_t s);
cudaError_t launch_stem_wgrad(const CUtensorMap& mapDy, const CUtensorMap& mapXs, const GemmParams& p, int grid,
                              cudaStream_t s);
cudaError_t launch_gemm_halo(const CUtensorMap& mapA, const CUtensorMap& mapB, const CUtensorMap& mapC,
                             const GemmParams& p, int grid, cudaStream_t stream);
// Wide halo engine (pf16_halo.cu): 3x3 / stride 1 / pad 1 forward convolutions with
// BN = 128 or 256 output channels (one N tile) over p.halo_chunks 64-channel
// input chunks.  mapA: 4-D tiled map over the input, dims (c, w, h, n) with
// boxes (64, halo_ws, halo_box_rows, 1) when halo_ipr = 1, or (c, w, n, h)
// with boxes (64, 16, 4, halo_box_rows) when four images of halo_wi = 16
// columns share a padded row; mapB: weights [BN][9 * Cin] (LD_TILED_K, boxes
// 64 x BN); mapC:
// 4-D map over the output, (c, w, h, n) with boxes (64, 32, 1, 1) or
// (c, w, n, h) with boxes (64, 16, 2, 1).  p.m_tiles tiles of 128 padded-grid
// rows; forward statistics (optional) as k_gemm's plain epilogue.
cudaError_t launch_gemm_halo_wide(int BN, const CUtensorMap& mapA, const CUtensorMap& mapB, const CUtensorMap& mapC,
                                  const GemmParams& p, int grid, cudaStream_t stream);
// Wide halo weight gradient (pf16_halo.cu): 3x3 / stride 1 / pad 1 with
// p.M = K output channels (a multiple of 128) and p.halo_chunks 64-channel
// input chunks.  mDy / mX: 4-D tiled maps (c, w, n, h) over dy [N][H][W][K]
// and x [N][H][W][C], boxes (64, halo_wi, halo_ipr, 1) with halo_wi = W + 1
// (halo_w = W, halo_h = H).  p.num_kb tiles (image group g, row h at tile
// g * H + h) in p.splits chunks of p.kb_per_split; p.m_tiles = p.splits x
// 3 x halo_chunks x K / 128 units; chunk q's partial plane at p.out + q * K *
// p.ldo (p.ldo = 9 * C), laid out as dw.
cudaError_t launch_wgrad3x3_wide(const CUtensorMap& mDy, const CUtensorMap& mX, const GemmParams& p, int grid,
                                 cudaStream_t stream);

// ---------------------------------------------------------------------------
// Memory-bound kernels (pf16_elementwise.cu).  All return cudaError_t of the
// launch.
// ---------------------------------------------------------------------------
cudaError_t launch_sgd(uint16_t* w, uint16_t* v, const uint16_t* g, size_t n, uint16_t lr,
                       uint16_t mom, uint16_t wd, cudaStream_t s);
// one thread waits (bounded by limit_ns) for *flag == value; expiry records
// PF16_ERR_TIMEOUT in *status.  A plain launch: it starts after its predecessor.
cudaError_t launch_wait_flag(const uint32_t* flag, uint32_t value, unsigned long long limit_ns, int* status,
                             cudaStream_t s);
// sum of `splits` FP16 partial matrices [splits][rows][cols] by a balanced
// pairwise tree; the result row r goes to out + r*ldo (only cols_out columns).
// Data-parallel exchange, combining step (pf16_allreduce_combine): n and
// plane_stride multiples of 8, 1 <= world <= 1024.
cudaError_t launch_dp_combine(const uint16_t* planes, int world, size_t n, size_t plane_stride, uint16_t scale,
                              uint16_t* out, cudaStream_t s);
cudaError_t launch_splitk_reduce(const uint16_t* parts, int splits, long long rows, int cols,
                                 uint16_t* out, long long ldo, int cols_out, cudaStream_t s);
// stem patches: col[m][j] = x[n, 2p+r-3, 2q+s-3, c] for j = (r*7+s)*3+c < 147, 0 up to kcol.
cudaError_t launch_stem_im2col(const uint16_t* x, uint16_t* col, int N, int H, int W, int P,
                               int Q, int R, int S, int C, int stride, int pad, int kcol,
                               cudaStream_t s);
// stem space-to-depth: xs = N x Hs x Ws x 16 and the 64 x 256 packed filter wsd
// of the 4x4 stride-1 form of the 7x7 / stride 2 / pad 3 convolution
cudaError_t launch_stem_s2d(const uint16_t* x, const uint16_t* w, uint16_t* xs, uint16_t* wsd, int N, int H,
                            int W, int Hs, int Ws, int K, cudaStream_t s);
// dw[k][r][s][c] (7 x 7 x 3) from the stem weight gradient's reduced 128 x 128
// [(a, k)][(u/2, v, ch)] matrix
cudaError_t launch_stem_wgrad_scatter(const uint16_t* dws, uint16_t* dw, int K, cudaStream_t s);
// w[K][kin] -> wpad[K][kcol] (zero padded)
cudaError_t launch_pad_rows(const uint16_t* w, uint16_t* wpad, int K, int kin, int kcol,
                            cudaStream_t s);
// zero the positions of a strided output no stride phase reaches (or all)
cudaError_t launch_fill_zero(uint16_t* p, size_t n, cudaStream_t s);

// Statistics grid of one direction: CTA b owns row chunks b, b + blocks, ...
struct BnPlan {
  int blocks;
  int chunks_per_cta;     // most chunks one CTA owns
  int blocks_pow2;
};
struct BnLaunch {
  int R, C;
  uint16_t eps, post_scale;
  int relu, residual;
  int swap;               // PF16_BN_SWAP: gamma * (s * xhat + residual) + beta
  int chunk_rows;         // rows per statistics chunk (contiguous in memory)
  BnPlan fwd, bwd;
  int* status;            // device status word (bounded waits record timeouts here)
};
// relu_mask (optional, ReLU only): one bit per element, byte [row][c/8].
cudaError_t launch_bn_fwd(const BnLaunch& b, const uint16_t* x, const uint16_t* gamma,
                          const uint16_t* beta, const uint16_t* residual, uint16_t* y,
                          uint8_t* relu_mask, uint16_t* mean, uint16_t* invstd, uint16_t* ws,
                          cudaStream_t s);
// Forward from conv-output statistics (pf16_conv_fwd_bnstats): final + apply.
cudaError_t launch_bn_fwd_given_stats(const BnLaunch& b, const uint8_t* conv_stats, const uint16_t* x,
                                      const uint16_t* gamma, const uint16_t* beta,
                                      const uint16_t* residual, uint16_t* y, uint8_t* relu_mask,
                                      uint16_t* mean, uint16_t* invstd, cudaStream_t s);
// The stem's BatchNorm + ReLU + 3x3 / stride 2 / pad 1 max pooling (x is
// N x H x W x C; pooled and codes N x P x Q x C, P = (H - 1) / 2 + 1): the
// statistics as launch_bn_fwd(_given_stats), then one fused pass.
int bn_pool_smem_bytes(int W, int C);
cudaError_t launch_bn_relu_pool_fwd(const BnLaunch& b, const uint8_t* conv_stats, const uint16_t* x,
                                    const uint16_t* gamma, const uint16_t* beta, uint16_t* mean,
                                    uint16_t* invstd, uint16_t* pooled, uint8_t* codes, uint8_t* mask,
                                    uint16_t* ws, int N, int H, int W, cudaStream_t s);
// ReLU decisions from relu_mask when non-null, else from y_saved.
cudaError_t launch_bn_bwd(const BnLaunch& b, const uint16_t* x, const uint16_t* gamma,
                          const uint16_t* mean, const uint16_t* invstd, const uint16_t* dy,
                          const uint16_t* y_saved, const uint8_t* relu_mask, uint16_t* dx,
                          uint16_t* dgamma, uint16_t* dbeta, uint16_t* dres, uint16_t* ws,
                          cudaStream_t s, const uint8_t* dgrad_stats = nullptr,
                          const uint16_t* residual = nullptr);
void bn_plan(int R, int C, BnLaunch* b);
size_t bn_ws_bytes(const BnLaunch& b);

// codes (optional): per output element the window position r*3+s of its first maximum
cudaError_t launch_maxpool_fwd(const uint16_t* x, uint16_t* y, uint8_t* codes, int N, int H, int W,
                               int C, cudaStream_t s);
cudaError_t launch_maxpool_bwd_codes(const uint8_t* codes, const uint16_t* dy, uint16_t* dx, int N,
                                     int H, int W, int C, cudaStream_t s);
cudaError_t launch_maxpool_bwd(const uint16_t* x, const uint16_t* dy, uint16_t* dx, int N, int H,
                               int W, int C, cudaStream_t s);
cudaError_t launch_avgpool_fwd(const uint16_t* x, uint16_t* y, int N, int HW, int C,
                               cudaStream_t s);
cudaError_t launch_avgpool_bwd(const uint16_t* dy, uint16_t* dx, int N, int HW, int C,
                               cudaStream_t s);
cudaError_t launch_softmax_xent(const uint16_t* logits, const uint16_t* bias,
                                const int32_t* labels, int B, int K, uint16_t* loss,
                                uint16_t* dlogits, uint16_t* dbias, uint16_t* ws,
                                cudaStream_t s);

}  // namespace pf16
