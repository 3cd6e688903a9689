// C-ABI of libpf16 (declared in include/pf16.h): argument validation, the
// per-call plan of each convolution pass (tile width, split-K, stride phases),
// TMA tensor-map encoding and kernel dispatch.  Nothing here allocates device
// memory; every call is asynchronous on the caller's stream.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "../../include/pf16.h"
#include "pf16_internal.h"
#include "pf16_ptx.cuh"

namespace pf16 {

// Device status word: bounded device waits that expire record PF16_ERR_TIMEOUT here.
__device__ int g_pf16_status = 0;

namespace {

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
typedef CUresult (*EncodeIm2colFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const int*, const int*,
                                   cuuint32_t, cuuint32_t, const cuuint32_t*,
                                   CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

std::once_flag g_fn_once;
EncodeTiledFn g_encode_tiled = nullptr;
EncodeIm2colFn g_encode_im2col = nullptr;

bool driver_fns() {
  std::call_once(g_fn_once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode_tiled = reinterpret_cast<EncodeTiledFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeIm2col", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode_im2col = reinterpret_cast<EncodeIm2colFn>(p);
  });
  return g_encode_tiled && g_encode_im2col;
}

constexpr int kMaxDevices = 64;
std::mutex g_dev_mu;
int* g_status_ptr[kMaxDevices] = {nullptr};
int g_num_sms[kMaxDevices] = {0};

// Per-device constants: status-word address and SM count.
int device_consts(int** status, int* sms) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return PF16_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_dev_mu);
  if (!g_status_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_pf16_status) != cudaSuccess) return PF16_ERR_CUDA;
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return PF16_ERR_CUDA;
    g_status_ptr[dev] = static_cast<int*>(p);
    g_num_sms[dev] = n;
  }
  *status = g_status_ptr[dev];
  *sms = g_num_sms[dev];
  return PF16_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
size_t round_up(size_t v, size_t a) { return (v + a - 1) / a * a; }
int cdiv(long long a, long long b) { return (int)((a + b - 1) / b); }

// 2-D tiled map over a row-major [rows][cols] FP16 matrix with row stride ld (elements).
bool map_2d(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, uint64_t ld,
            uint32_t box_cols, uint32_t box_rows,
            CUtensorMapSwizzle swz = CU_TENSOR_MAP_SWIZZLE_128B) {
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {ld * 2};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t es[2] = {1, 1};
  return g_encode_tiled(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(base), dims,
                        strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 3-D tiled map: dims (d0 contiguous, d1, d2) with byte strides s1, s2.
bool map_3d(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint64_t s1,
            uint64_t s2, uint32_t b0, uint32_t b1, uint32_t b2) {
  cuuint64_t dims[3] = {d0, d1, d2};
  cuuint64_t strides[2] = {s1, s2};
  cuuint32_t box[3] = {b0, b1, b2};
  cuuint32_t es[3] = {1, 1, 1};
  return g_encode_tiled(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, const_cast<void*>(base), dims,
                        strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// im2col map over an NHWC tensor.  The bounding box of filter-corner positions
// starts at (lo_h, lo_w) and holds gh x gw points at `step`; each load yields
// `pixels` consecutive grid points x 64 channels.
bool map_im2col(CUtensorMap* m, const void* base, int N, int H, int W, int C, int lo_h, int lo_w,
                int gh, int gw, int step, int pixels) {
  const int up_h = lo_h + (gh - 1) * step - (H - 1);
  const int up_w = lo_w + (gw - 1) * step - (W - 1);
  if (lo_h < -128 || lo_h > 127 || lo_w < -128 || lo_w > 127 || up_h < -128 || up_h > 127 ||
      up_w < -128 || up_w > 127)
    return false;
  cuuint64_t dims[4] = {(cuuint64_t)C, (cuuint64_t)W, (cuuint64_t)H, (cuuint64_t)N};
  cuuint64_t strides[3] = {(cuuint64_t)C * 2, (cuuint64_t)W * C * 2, (cuuint64_t)H * W * C * 2};
  int lower[2] = {lo_w, lo_h};
  int upper[2] = {up_w, up_h};
  cuuint32_t es[4] = {1, (cuuint32_t)step, (cuuint32_t)step, 1};
  return g_encode_im2col(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<void*>(base), dims,
                         strides, lower, upper, 64, (cuuint32_t)pixels, es,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                         CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// ---------------------------------------------------------------- conv plans
enum ConvKind { KIND_GENERIC = 0, KIND_STEM = 1, KIND_FC = 2 };

struct Shape {
  long long N, H, W, C, K, R, S, st, pad, P, Q;
  ConvKind kind;
};

int conv_shape(const pf16_conv_desc* d, Shape* s) {
  if (!d) return PF16_ERR_NULL;
  if (d->n <= 0 || d->h <= 0 || d->w <= 0 || d->c <= 0 || d->k <= 0 || d->r <= 0 || d->s <= 0 ||
      d->pad < 0 || d->stride <= 0)
    return PF16_ERR_SHAPE;
  if (d->stride > 2 || d->r > 7 || d->s > 7 || d->pad >= std::max(d->r, d->s))
    return PF16_ERR_UNSUPPORTED;
  s->N = d->n;
  s->H = d->h;
  s->W = d->w;
  s->C = d->c;
  s->K = d->k;
  s->R = d->r;
  s->S = d->s;
  s->st = d->stride;
  s->pad = d->pad;
  if (d->h + 2 * d->pad < d->r || d->w + 2 * d->pad < d->s) return PF16_ERR_SHAPE;
  s->P = (d->h + 2 * d->pad - d->r) / d->stride + 1;
  s->Q = (d->w + 2 * d->pad - d->s) / d->stride + 1;
  const long long lim = (1ll << 31) - 1;
  if (s->N * s->H * s->W * s->C > lim * 8 || s->N * s->P * s->Q > lim / 2 ||
      s->N * s->H * s->W > lim / 2 || s->K * s->R * s->S * s->C > lim)
    return PF16_ERR_SHAPE;
  if (d->c == 3) {
    if (d->k % 64 != 0) return PF16_ERR_UNSUPPORTED;
    // the patch gather stages r padded input rows in shared memory
    if ((long long)d->r * (d->w + 2 * d->pad) * 3 * 2 > 200 * 1024) return PF16_ERR_UNSUPPORTED;
    s->kind = KIND_STEM;
  } else if (d->h == 1 && d->w == 1 && d->r == 1 && d->s == 1 && d->pad == 0 && d->stride == 1) {
    if (d->c % 64 != 0 || d->k % 8 != 0) return PF16_ERR_UNSUPPORTED;
    s->kind = KIND_FC;
  } else {
    if (d->c % 64 != 0 || d->k % 64 != 0) return PF16_ERR_UNSUPPORTED;
    s->kind = KIND_GENERIC;
  }
  return PF16_OK;
}

int pick_bn_out(long long n) {  // tile width for an output of n columns
  if (n <= 64) return 64;
  if (n <= 128) return 128;
  if (n % 256 == 0 || n > 192) return 256;
  return 192;
}
int pick_bn_wgrad(long long n) {
  if (n % 256 == 0) return 256;
  if (n % 192 == 0) return 192;
  if (n % 128 == 0) return 128;
  if (n <= 64) return 64;
  return n <= 192 ? 192 : 256;
}

long long stem_kcol(const Shape& s) { return (long long)round_up((size_t)(s.R * s.S * s.C), 8); }

struct WgradSplit {
  int bn, m_tiles, n_tiles, num_kb, kb_per_split, splits;
  long long ncols;  // GEMM N
};

// Split-K plan of the weight gradient, independent of the device so that
// pf16_conv_workspace_size and the call always agree.  The persistent GEMM
// runs tiles * splits units on the 152 SMs of a GB300 in ceil(units / 152)
// rounds, so the split count is the one minimising a makespan model:
//   rounds * (K-blocks per split * t_kb + t_unit) + partial-plane traffic,
// with t_kb ~ 0.4 us per 128 x 256 x 64 block, t_unit ~ 1 us (pipeline fill
// and the partial tile's store) and the splits * |dw| FP16 partials written
// and read back at the reduce's effective ~2 TB/s (measured: a reduce call
// costs several microseconds beyond its bytes).  Between 4 and 64 K-blocks
// (4096 pixels) go into one FP16 tensor-memory accumulator; at most 1024
// splits.
constexpr int kPlanSms = 152;
constexpr double kPartialBw = 2e12;  // effective partial-plane bandwidth of the reduce, bytes/s

WgradSplit wgrad_split(const Shape& s) {
  WgradSplit w;
  w.ncols = s.kind == KIND_STEM ? stem_kcol(s) : s.R * s.S * s.C;
  w.bn = pick_bn_wgrad(w.ncols);
  w.m_tiles = cdiv(s.K, kBM);
  w.n_tiles = cdiv(w.ncols, w.bn);
  w.num_kb = cdiv(s.N * s.P * s.Q, kBK);
  const long long tiles = (long long)w.m_tiles * w.n_tiles;
  const double t_kb = 0.4e-6 * w.bn / 256.0, t_unit = 1.0e-6;
  const double dw_bytes = 2.0 * (double)s.K * (double)w.ncols;
  double best = -1.0;
  w.kb_per_split = std::min(w.num_kb, 64);
  w.splits = cdiv(w.num_kb, w.kb_per_split);
  for (int sp = 1; sp <= 1024; ++sp) {
    const int kps = cdiv(w.num_kb, sp);
    if (kps > 64) continue;
    if (kps < 4 && sp > 1) break;  // kps only shrinks from here
    const int real = cdiv(w.num_kb, kps);
    const long long rounds = (tiles * real + kPlanSms - 1) / kPlanSms;
    const double t = (double)rounds * (kps * t_kb + t_unit) + (real > 1 ? real * dw_bytes * 2.0 / kPartialBw : 0.0);
    if (best < 0.0 || t < best * (1.0 - 1e-9)) {
      best = t;
      w.kb_per_split = kps;
      w.splits = real;
    }
  }
  if (w.splits > 1024) {  // only when more than 65,536 K-blocks: fill 1024 splits
    w.kb_per_split = cdiv(w.num_kb, 1024);
    w.splits = cdiv(w.num_kb, w.kb_per_split);
  }
  return w;
}

// The ResNet stem (7x7, stride 2, pad 3, 3 -> 64 channels) runs as a 4x4
// stride-1 convolution over the 2x2 space-to-depth of its input: xs[n][I][J]
// holds 16 channels (a*2 + b)*4 + c = x[n][2I + a - 3][2J + b - 3][c] (c < 3;
// channel c = 3 and pixels outside x are 0), I < P + 3, J < Q + 3, and the
// 64 x 256 packed filter ws[k][(u*4 + v)*16 + (a*2 + b)*4 + c] =
// w[k][2u + a][2v + b][c] (0 where 2u + a or 2v + b reaches 7).  Returns the
// halo engine's padded row width, or 0 where the stem takes the patch GEMM.
int stem_s2d_width(const Shape& s, bool accum) {
  if (accum || s.kind != KIND_STEM || s.R != 7 || s.S != 7 || s.st != 2 || s.pad != 3 || s.K != 64)
    return 0;
  int ws = 0;
  if (s.Q + 3 <= 32 && s.P % 4 == 0)
    ws = 32;
  else if (s.Q + 3 <= 64 && s.P % 2 == 0)
    ws = 64;
  else if (s.Q + 3 <= 128)
    ws = 128;
  if (ws == 0 || (long long)s.N * s.P * ws / kBM > (1ll << 30)) return 0;
  return ws;
}
size_t stem_s2d_bytes(const Shape& s) { return round_up((size_t)(s.N * (s.P + 3) * (s.Q + 3) * 32), 256); }

// Stem weight gradient on the space-to-depth input (k_stem_wgrad): work units
// are the N * (P + 1) output rows (padded to 128 columns), accumulated in FP16
// over chunks of 32 rows (4,096 padded pixels) -- more only beyond 1,024
// chunks -- then summed by the split-K tree.  Workspace: xs, the chunks'
// 128 x 128 partials, the reduced 128 x 128 matrix.
struct StemWgradPlan {
  bool ok;
  long long rows;
  int per_chunk, chunks;
};
StemWgradPlan stem_wgrad_plan(const Shape& s) {
  StemWgradPlan w{false, 0, 0, 0};
  if (!stem_s2d_width(s, false)) return w;
  w.rows = s.N * (s.P + 1);
  w.per_chunk = 32;
  if (cdiv(w.rows, w.per_chunk) > 1024) w.per_chunk = (int)cdiv(w.rows, 1024);
  w.chunks = (int)cdiv(w.rows, w.per_chunk);
  w.ok = w.rows < (1ll << 30);
  return w;
}
size_t stem_wgrad_parts_bytes(const StemWgradPlan& w) { return round_up((size_t)w.chunks * 128 * 128 * 2, 256); }

// The 3x3 / stride 1 / pad 1 weight gradient with 64 input and 64 output
// channels on padded rows of 64 pixels (W + 2 <= 64): units of two output
// rows, at most 32 units (4,096 padded pixels) per FP16 accumulation and at
// most 1,024 chunks for the split-K tree.
struct Wgrad3Plan {
  bool ok;
  long long units;
  int per_chunk, chunks;
};
Wgrad3Plan wgrad3_plan(const Shape& s) {
  Wgrad3Plan w{false, 0, 0, 0};
  if (s.kind != KIND_GENERIC || s.R != 3 || s.S != 3 || s.st != 1 || s.pad != 1 || s.C != 64 || s.K != 64 ||
      s.W + 2 > 64)
    return w;
  w.units = s.N * ((s.P + 2) / 2);
  // as many rounds of 152 chunks (GB300's SM count) as 32-unit chunks need,
  // the units spread evenly over them
  const long long rounds = cdiv(w.units, 32ll * 152);
  w.per_chunk = (int)cdiv(w.units, rounds * 152);
  if (cdiv(w.units, w.per_chunk) > 1024) w.per_chunk = (int)cdiv(w.units, 1024);
  w.chunks = (int)cdiv(w.units, w.per_chunk);
  w.ok = w.units < (1ll << 30);
  return w;
}
size_t wgrad3_parts_bytes(const Wgrad3Plan& w) { return round_up((size_t)w.chunks * 64 * 576 * 2, 256); }

// The 3x3 / stride 1 / pad 1 weight gradient with K a multiple of 128 and C
// of 64 on the wide halo engine (k_wgrad3x3_wide): a tile is one image row
// of nb images of wi = W + 1 columns (at most 128 pixels), per_chunk tiles
// (at most 32: 4,096 pixels) per FP16 accumulation.  The chunk length
// minimises a makespan model on GB300's 152 SMs: rounds of units x chunk
// length x ~0.42 us per tile (8 MMAs of 128 x 192 x 16) plus the partial
// planes through the split-K tree at ~2 TB/s; at most 1,024 chunks.
struct WideWgradPlan {
  bool ok;
  int wi, nb, types, per_chunk, chunks;
  long long tiles;
};
WideWgradPlan wide_wgrad_plan(const Shape& s) {
  WideWgradPlan w{};
  if (s.kind != KIND_GENERIC || s.R != 3 || s.S != 3 || s.st != 1 || s.pad != 1 || s.K < 128 || s.K % 128 != 0 ||
      s.C % 64 != 0 || s.W + 1 > 128)
    return w;
  w.wi = (int)s.W + 1;
  w.nb = (int)std::min<long long>(128 / w.wi, s.N);
  w.tiles = cdiv(s.N, (long long)w.nb) * s.H;
  w.types = (int)(3 * (s.C / 64) * (s.K / 128));
  const double plane_us = (double)s.K * 9 * s.C * 2 / 2.0e6;
  double best = 1e300;
  for (int len = 1; len <= 32; ++len) {
    const long long chunks = cdiv(w.tiles, (long long)len);
    if (chunks > 1024) continue;
    const double t = (double)cdiv(chunks * w.types, 152ll) * len * 0.42 + (double)chunks * plane_us;
    if (t < best) {
      best = t;
      w.per_chunk = len;
      w.chunks = (int)chunks;
    }
  }
  w.ok = best < 1e300 && (long long)w.chunks * w.types < (1ll << 30);
  return w;
}
size_t wide_wgrad_parts_bytes(const Shape& s, const WideWgradPlan& w) {
  return round_up((size_t)w.chunks * s.K * 9 * s.C * 2, 256);
}

size_t ws_fwd(const Shape& s) {
  if (s.kind != KIND_STEM) return 0;
  const long long kc = stem_kcol(s);
  const size_t patch = round_up((size_t)(s.N * s.P * s.Q * kc * 2), 256) + round_up((size_t)(s.K * kc * 2), 256);
  // the space-to-depth route serves plain stores; PF16_ACCUMULATE takes the patch GEMM
  if (!stem_s2d_width(s, false)) return patch;
  return std::max(patch, stem_s2d_bytes(s) + (size_t)(s.K * 256 * 2));
}
size_t ws_wgrad(const Shape& s) {
  const StemWgradPlan sw = stem_wgrad_plan(s);
  if (sw.ok) return stem_s2d_bytes(s) + stem_wgrad_parts_bytes(sw) + 128 * 128 * 2;
  const Wgrad3Plan w3 = wgrad3_plan(s);
  if (w3.ok) return wgrad3_parts_bytes(w3);
  const WideWgradPlan ww = wide_wgrad_plan(s);
  if (ww.ok) return wide_wgrad_parts_bytes(s, ww);
  const WgradSplit w = wgrad_split(s);
  size_t b = 0;
  if (w.splits > 1 || s.kind == KIND_STEM) b += round_up((size_t)w.splits * s.K * w.ncols * 2, 256);
  if (s.kind == KIND_STEM) b += round_up((size_t)(s.N * s.P * s.Q * w.ncols * 2), 256);
  return b;
}

// Taps of one stride phase of the data gradient.  For output row h = st*i + ph
// the contributing filter rows r satisfy (ph + pad - r) % st == 0 and read dy
// row i + (ph + pad - r) / st; likewise for columns.
struct Phase {
  int gh, gw;           // output grid of the phase
  int nr, ns;           // contributing filter rows / columns
  int rr[7], ar[7];     // filter row and dy-row offset
  int ss[7], bs[7];     // filter column and dy-column offset
  bool empty() const { return nr == 0 || ns == 0 || gh <= 0 || gw <= 0; }
};

Phase make_phase(const Shape& s, int ph, int pw) {
  Phase f;
  f.gh = (int)((s.H - ph + s.st - 1) / s.st);
  f.gw = (int)((s.W - pw + s.st - 1) / s.st);
  f.nr = f.ns = 0;
  for (int r = 0; r < s.R; ++r) {
    const long long t = ph + s.pad - r;
    if (((t % s.st) + s.st) % s.st == 0) {
      f.rr[f.nr] = r;
      f.ar[f.nr++] = (int)(t >= 0 ? t / s.st : -((-t) / s.st));
    }
  }
  for (int c = 0; c < s.S; ++c) {
    const long long t = pw + s.pad - c;
    if (((t % s.st) + s.st) % s.st == 0) {
      f.ss[f.ns] = c;
      f.bs[f.ns++] = (int)(t >= 0 ? t / s.st : -((-t) / s.st));
    }
  }
  return f;
}

void set_kmajor(GemmParams& p, bool a, bool b) {
  if (a) {
    p.a_lbo = 16;
    p.a_sbo = 1024;
    p.a_kstep = 32;
  }
  if (b) {
    p.b_lbo = 16;
    p.b_sbo = 1024;
    p.b_kstep = 32;
  }
}
void set_mnmajor(GemmParams& p, bool a, bool b) {
  if (a) {
    p.a_lbo = 8192;
    p.a_sbo = 1024;
    p.a_kstep = 2048;
  }
  if (b) {
    p.b_lbo = 8192;
    p.b_sbo = 1024;
    p.b_kstep = 2048;
  }
}

GemmParams base_params(int* status) {
  GemmParams p;
  memset(&p, 0, sizeof(p));
  p.kb_per_split = 1 << 30;
  p.splits = 1;
  p.status = status;
  p.wait_limit_ns = 4000000000ull;
  return p;
}

// Levels of an epilogue warp's padded tile tree (backward statistics): `ctas`
// CTAs share `units` tiles round robin, and each CTA's two
// epilogue groups take alternate tiles.
int tile_tree_levels(long long units, long long ctas) {
  const long long per_cta = (units + ctas - 1) / ctas;
  const long long per_group = (per_cta + 1) / 2;
  int l = 0;
  while ((1ll << l) < per_group) ++l;
  return l;
}

int run(int BN, const CUtensorMap& a, const CUtensorMap& b, GemmParams& p, int sms,
        cudaStream_t st) {
  p.m_tiles = cdiv(p.M, kBM);
  p.n_tiles = cdiv(p.N, BN);
  if (p.splits == 1) p.kb_per_split = p.num_kb;
  p.idesc = idesc_f16(kBM, BN, p.a_mode == LD_TILED_MN,
                      p.b_mode == LD_TILED_MN || p.b_mode == LD_IM2COL_MN || p.b_mode == LD_TAP3D_MN,
                      p.d_f32 != 0);
  const long long units = (long long)p.m_tiles * p.n_tiles * p.splits;
  if (units <= 0 || p.num_kb <= 0) return PF16_OK;
  // Row-major outputs leave through TMA stores of 32-row x 64-column boxes
  // (PF16_ACCUMULATE through TMA reduce-add stores, out = rn(out + tile)); the
  // split-K partials use a 3-D map so each split's plane is clipped on its own.
  CUtensorMap c = a;
  p.tma_store = 0;
  if ((p.out_mode == OUT_STORE || p.out_mode == OUT_ACCUM) && !p.remap) {
    if (!map_2d(&c, p.out, p.N, p.M, p.ldo, 64, 32)) return PF16_ERR_CUDA;
    p.tma_store = 1;
  } else if (p.out_mode == OUT_PARTIAL) {
    if (!map_3d(&c, p.out, p.N, p.M, p.splits, p.ldo * 2, (uint64_t)p.M * p.ldo * 2, 64, 32, 1))
      return PF16_ERR_CUDA;
    p.tma_store = 1;
  }
  // backward statistics: the BatchNorm input (and the addend) enter the
  // epilogue as TMA tiles of the output's 32 x 64 boxes
  // (remapped rows -- a stride phase -- read it by plain loads instead)
  CUtensorMap mx = c, md = c;
  if (p.bs_x) {
    if (p.out_mode != OUT_STORE) return PF16_ERR_UNSUPPORTED;
    if (p.remap) {
      if (p.add_src) return PF16_ERR_UNSUPPORTED;
    } else {
      if (!p.tma_store) return PF16_ERR_UNSUPPORTED;
      if (!map_2d(&mx, p.bs_x, p.N, p.M, p.ldo, 64, 32)) return PF16_ERR_CUDA;
      if (p.add_src && !map_2d(&md, p.add_src, p.N, p.M, p.ldo, 64, 32)) return PF16_ERR_CUDA;
    }
  }
  int grid = (int)std::min<long long>(units, sms);
  if (p.st_mean) {
    // fused statistics: every CTA keeps one n-tile (grid a multiple of n_tiles), at most
    // kBnStatSlots CTAs (one statistics slot each) per n-tile
    grid = std::min(grid, kBnStatSlots * p.n_tiles);
    grid -= grid % p.n_tiles;
    if (p.bs_x && (p.bs_levels = tile_tree_levels(units, grid)) >= kMaxTileTreeLevels) return PF16_ERR_UNSUPPORTED;
  }
  return launch_gemm(BN, a, b, c, p, grid, st, &mx, &md) == cudaSuccess ? PF16_OK : PF16_ERR_CUDA;
}

// Point the GEMM's fused statistics at the BatchNorm backward sources.
void set_bwd_stats(GemmParams& p, const pf16_bn_source* bn) {
  if (!bn) return;
  p.bs_x = bn->x;
  p.bs_mask = bn->relu_mask;
  p.bs_mean = bn->mean;
  p.bs_invstd = bn->invstd;
}

// Point the GEMM's fused statistics at a conv-output statistics buffer of C channels.
void set_stats(GemmParams& p, void* stats, long long C) {
  if (!stats) return;
  uint8_t* b = static_cast<uint8_t*>(stats);
  p.st_hdr = reinterpret_cast<int*>(b);
  p.st_mean = reinterpret_cast<uint16_t*>(b + bnstat_off_mean());
  p.st_var = reinterpret_cast<uint16_t*>(b + bnstat_off_var(C));
  p.st_cnt = reinterpret_cast<int*>(b + bnstat_off_cnt(C));
}

// Every stride phase of a stride-2 data gradient in one launch, when the four
// phases share their output grid and im2col origin (even H and W with the
// usual padding: the ResNet layers) and reach every position.  The units are
// ordered by phase, the phases by falling tap count, so that the round-robin
// schedule ends on the shortest tiles.  PF16_ERR_UNSUPPORTED: the phases
// differ; the caller launches them one by one.
bool phases_one_launch(const Shape& s, Phase* f = nullptr) {
  Phase g[4];
  if (!f) f = g;
  if (s.kind == KIND_STEM || s.st != 2 || (s.R == 1 && s.S == 1)) return false;
  int taps = 0;
  for (int q = 0; q < 4; ++q) {
    f[q] = make_phase(s, q >> 1, q & 1);
    if (f[q].empty()) return false;
    taps += f[q].nr * f[q].ns;
  }
  if (taps > kMaxTaps) return false;
  const int amin = *std::min_element(f[0].ar, f[0].ar + f[0].nr), bmin = *std::min_element(f[0].bs, f[0].bs + f[0].ns);
  for (int q = 1; q < 4; ++q) {
    const int a = *std::min_element(f[q].ar, f[q].ar + f[q].nr), b = *std::min_element(f[q].bs, f[q].bs + f[q].ns);
    if (f[q].gh != f[0].gh || f[q].gw != f[0].gw || a != amin || b != bmin) return false;
  }
  return true;
}

int run_dgrad_phases(const Shape& s, const uint16_t* dy, const uint16_t* w, uint16_t* dx, int* status, int sms,
                     cudaStream_t st, bool f32, bool accum, int BN, void* stats = nullptr,
                     const pf16_bn_source* bn = nullptr) {
  Phase f[4];
  int order[4] = {0, 1, 2, 3};
  if (!phases_one_launch(s, f)) return PF16_ERR_UNSUPPORTED;
  const int amin = *std::min_element(f[0].ar, f[0].ar + f[0].nr), bmin = *std::min_element(f[0].bs, f[0].bs + f[0].ns);
  std::stable_sort(order, order + 4, [&](int x, int y) { return f[x].nr * f[x].ns > f[y].nr * f[y].ns; });
  const int gh = f[0].gh, gw = f[0].gw;
  GemmParams p = base_params(status);
  p.d_f32 = f32 ? 1 : 0;
  set_stats(p, stats, s.C);  // the four phases together cover every pixel once
  if (stats) set_bwd_stats(p, bn);
  CUtensorMap ma, mb;
  p.M = (int)(s.N * gh * gw);
  p.N = (int)s.C;
  p.a_mode = LD_IM2COL_K;
  p.b_mode = LD_TAP3D_MN;
  set_kmajor(p, true, false);
  set_mnmajor(p, false, true);
  p.ga = PixGrid{gh, gw, 1, amin, bmin};
  if (!map_im2col(&ma, dy, (int)s.N, (int)s.P, (int)s.Q, (int)s.K, amin, bmin, gh, gw, 1, kBM))
    return PF16_ERR_CUDA;
  if (!map_3d(&mb, w, s.C, s.R * s.S, s.K, s.C * 2, s.R * s.S * s.C * 2, 64, 1, 64)) return PF16_ERR_CUDA;
  p.a_cpt = p.b_cpt = (int)(s.K / 64);
  int t = 0;
  for (int k = 0; k < 4; ++k) {
    const Phase& g = f[order[k]];
    p.ph_kb[k] = t * p.a_cpt;
    p.ph_h[k] = (int8_t)(order[k] >> 1);
    p.ph_w[k] = (int8_t)(order[k] & 1);
    for (int i = 0; i < g.nr; ++i)
      for (int j = 0; j < g.ns; ++j, ++t) {
        p.tap_dr[t] = (int8_t)(g.ar[i] - amin);
        p.tap_ds[t] = (int8_t)(g.bs[j] - bmin);
        p.tap_w[t] = (int8_t)(g.rr[i] * s.S + g.ss[j]);
      }
  }
  p.ph_kb[4] = t * p.a_cpt;
  p.ntaps = t;
  p.num_kb = p.ph_kb[4];
  p.nphase = 4;
  p.splits = 4;
  p.out = dx;
  p.ldo = s.C;
  p.out_mode = accum ? OUT_ACCUM : OUT_STORE;
  p.remap = 1;
  p.rm_gh = gh;
  p.rm_gw = gw;
  p.rm_H = (int)s.H;
  p.rm_W = (int)s.W;
  p.rm_step = 2;
  return run(BN, ma, mb, p, sms, st);
}

int check_common(const void* a, const void* b, const void* c) {
  if (!a || !b || !c) return PF16_ERR_NULL;
  if (!aligned16(a) || !aligned16(b) || !aligned16(c)) return PF16_ERR_ALIGN;
  return PF16_OK;
}

}  // namespace
}  // namespace pf16

using namespace pf16;

extern "C" {

size_t pf16_conv_workspace_size(const pf16_conv_desc* d, int pass) {
  Shape s;
  if (conv_shape(d, &s) != PF16_OK) return 0;
  if (pass == PF16_PASS_FWD) return ws_fwd(s);
  if (pass == PF16_PASS_DGRAD) return 0;
  if (pass == PF16_PASS_WGRAD) return ws_wgrad(s);
  return 0;
}

// Padded row width of the halo engine for a 3x3 / stride 1 / pad 1 layer with
// 64 input and 64 output channels, or 0 where it does not apply: the padded
// grid needs ws >= W + 2 and a 128-row tile of 128 / ws whole image rows that
// never straddles two images.
int halo_width(const Shape& s, bool accum) {
  if (accum || s.kind != KIND_GENERIC || s.R != 3 || s.S != 3 || s.st != 1 || s.pad != 1) return 0;
  if (s.C != 64 || s.K != 64) return 0;
  const int ws = s.W + 2 <= 32 ? 32 : (s.W + 2 <= 64 ? 64 : 0);
  if (ws == 0 || s.H % (kBM / ws) != 0) return 0;
  if ((long long)s.N * s.H * ws / kBM > (1ll << 30)) return 0;
  return ws;
}

// 3x3 stride-1 forward (dgrad = false: in = x, weights [K][9*C]) or data
// gradient (dgrad = true: in = dy, weights viewed (C, 9, K), taps flipped)
// through the halo engine.  in and out are N x H x W x 64.
int run_halo(const Shape& s, int ws, bool dgrad, const uint16_t* in, const uint16_t* w, uint16_t* out,
             int* status, int sms, cudaStream_t st, bool f32, void* stats = nullptr,
             const pf16_bn_source* bn = nullptr) {
  GemmParams p = base_params(status);
  p.d_f32 = f32 ? 1 : 0;
  set_stats(p, stats, 64);
  set_bwd_stats(p, bn);
  CUtensorMap ma, mb, mc;
  const long long N = s.N, H = s.H, W = s.W;
  cuuint64_t dims[4] = {64, (cuuint64_t)W, (cuuint64_t)H, (cuuint64_t)N};
  cuuint64_t strides[3] = {128, (cuuint64_t)W * 128, (cuuint64_t)(H * W * 128)};
  cuuint32_t box[4] = {64, (cuuint32_t)ws, (cuuint32_t)(kBM / ws + 2), 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  if (g_encode_tiled(&ma, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<uint16_t*>(in), dims, strides,
                     box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return PF16_ERR_CUDA;
  if (!map_3d(&mc, out, 64, W, N * H, 128, W * 128, 64, 32, 1)) return PF16_ERR_CUDA;
  p.ntaps = 9;
  for (int t = 0; t < 9; ++t) {
    p.tap_dr[t] = (int8_t)(t / 3);
    p.tap_ds[t] = (int8_t)(t % 3);
    p.tap_w[t] = (int8_t)(dgrad ? 8 - t : t);  // the data gradient reads the filter flipped
  }
  if (dgrad) {
    p.b_mode = LD_TAP3D_MN;
    set_mnmajor(p, false, true);
    if (!map_3d(&mb, w, 64, 9, 64, 128, 9 * 128, 64, 1, 64)) return PF16_ERR_CUDA;
  } else {
    p.b_mode = LD_TILED_K;
    set_kmajor(p, false, true);
    if (!map_2d(&mb, w, 9 * 64, 64, 9 * 64, 64, 64)) return PF16_ERR_CUDA;
  }
  // N = 192: the slices of taps (r, 0..2), contiguous in shared memory
  p.idesc = idesc_f16(kBM, 192, false, dgrad, f32);
  p.halo_ws = ws;
  p.halo_h = (int)H;
  p.halo_w = (int)W;
  p.halo_cb = 128;
  p.halo_box_rows = kBM / ws + 2;
  p.halo_row0 = -1;
  p.halo_col0 = -1;
  p.N = 64;
  p.ldo = 64;
  p.n_tiles = 1;
  p.m_tiles = (int)(N * H * ws / kBM);
  int grid = p.m_tiles < sms ? p.m_tiles : sms;
  if (stats && grid > kBnStatSlots) grid = kBnStatSlots;
  if (p.bs_x && (p.bs_levels = tile_tree_levels(p.m_tiles, grid)) >= kMaxTileTreeLevels) return PF16_ERR_UNSUPPORTED;
  return launch_gemm_halo(ma, mb, mc, p, grid, st) == cudaSuccess ? PF16_OK : PF16_ERR_CUDA;
}

// Layout of the wide halo engine (pf16_halo.cu) for a 3x3 / stride 1 / pad 1
// layer with cin input and cout output channels (cout 128 or 256, cin a
// multiple of 64), or ipr = 0 where it does not apply: one image per padded
// row of ws = 32 or 64 columns (at least W + 2; the tile's 128 / ws rows must
// divide H), or four images of wi = 16 columns side by side (W <= 14, two rows
// per tile dividing H, N a multiple of 4), whichever wastes fewer padding
// columns, and only when at least three quarters of the columns are pixels.
struct WidePlan {
  int ipr, wi, ws;
};
WidePlan halo_wide_plan(const Shape& s, long long cin, long long cout, bool accum) {
  WidePlan best{0, 0, 0};
  if (accum || s.kind != KIND_GENERIC || s.R != 3 || s.S != 3 || s.st != 1 || s.pad != 1) return best;
  if (cin % 64 != 0 || (cout != 128 && cout != 256)) return best;
  double eff = 0.0;
  for (int ws : {32, 64})
    if (s.W + 2 <= ws && s.H % (kBM / ws) == 0 && (double)s.W / ws > eff) {
      eff = (double)s.W / ws;
      best = WidePlan{1, ws, ws};
    }
  if (s.W + 2 <= 16 && s.H % 2 == 0 && s.N % 4 == 0 && (double)s.W / 16 > eff) {
    eff = (double)s.W / 16;
    best = WidePlan{4, 16, 64};
  }
  if (eff < 0.75) best = WidePlan{0, 0, 0};
  return best;
}

// 3x3 stride-1 forward through the wide halo engine: in = x [N,H,W,C],
// weights [K][9*C], out = y [N,H,W,K].  (The data gradients keep the im2col
// GEMM: with their fused backward statistics, which every 3x3 data gradient of
// the training step takes, the wide engine measured no faster -- 28x28, 128
// channels: 103 against 95 us at batch 256 -- its MMAs then sharing the SM
// with the epilogue's loads and trees; and the plain call must give the same
// bits as the one with statistics.)
int run_halo_wide(const Shape& s, const WidePlan& wp, const uint16_t* in, const uint16_t* w, uint16_t* out,
                  int* status, int sms, cudaStream_t st, bool f32, void* stats = nullptr) {
  const long long cin = s.C, cout = s.K;
  const long long N = s.N, H = s.H, W = s.W;
  const int rpt = kBM / wp.ws;
  GemmParams p = base_params(status);
  p.d_f32 = f32 ? 1 : 0;
  set_stats(p, stats, cout);
  CUtensorMap ma, mb, mc;
  cuuint32_t es[4] = {1, 1, 1, 1};
  {
    const cuuint64_t pix = (cuuint64_t)cin * 2, row = (cuuint64_t)W * pix, img = (cuuint64_t)H * row;
    const bool one = wp.ipr == 1;
    cuuint64_t dims[4] = {(cuuint64_t)cin, (cuuint64_t)W, (cuuint64_t)(one ? H : N), (cuuint64_t)(one ? N : H)};
    cuuint64_t strides[3] = {pix, one ? row : img, one ? img : row};
    cuuint32_t box[4] = {64, (cuuint32_t)wp.wi, (cuuint32_t)(one ? rpt + 2 : wp.ipr), (cuuint32_t)(one ? 1 : rpt + 2)};
    if (g_encode_tiled(&ma, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<uint16_t*>(in), dims, strides, box, es,
                       CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                       CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return PF16_ERR_CUDA;
  }
  {
    const cuuint64_t pix = (cuuint64_t)cout * 2, row = (cuuint64_t)W * pix, img = (cuuint64_t)H * row;
    const bool one = wp.ipr == 1;
    cuuint64_t dims[4] = {(cuuint64_t)cout, (cuuint64_t)W, (cuuint64_t)(one ? H : N), (cuuint64_t)(one ? N : H)};
    cuuint64_t strides[3] = {pix, one ? row : img, one ? img : row};
    cuuint32_t box[4] = {64, (cuuint32_t)(one ? 32 : 16), (cuuint32_t)(one ? 1 : 2), 1};
    if (g_encode_tiled(&mc, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, out, dims, strides, box, es,
                       CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                       CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return PF16_ERR_CUDA;
  }
  p.ntaps = 9;
  for (int t = 0; t < 9; ++t) {
    p.tap_dr[t] = (int8_t)(t / 3);
    p.tap_ds[t] = (int8_t)(t % 3);
    p.tap_w[t] = (int8_t)t;
  }
  p.b_mode = LD_TILED_K;
  set_kmajor(p, false, true);
  if (!map_2d(&mb, w, 9 * cin, cout, 9 * cin, 64, (uint32_t)cout)) return PF16_ERR_CUDA;
  p.idesc = idesc_f16(kBM, (int)cout, false, false, f32);
  p.halo_ws = wp.ws;
  p.halo_ipr = wp.ipr;
  p.halo_wi = wp.wi;
  p.halo_h = (int)H;
  p.halo_w = (int)W;
  p.halo_box_rows = rpt + 2;
  p.halo_chunks = (int)(cin / 64);
  p.N = (int)cout;
  p.ldo = cout;
  p.n_tiles = 1;
  p.m_tiles = (int)((N / wp.ipr) * (H / rpt));
  int grid = p.m_tiles < sms ? p.m_tiles : sms;
  if (stats && grid > kBnStatSlots) grid = kBnStatSlots;
  return launch_gemm_halo_wide((int)cout, ma, mb, mc, p, grid, st) == cudaSuccess ? PF16_OK : PF16_ERR_CUDA;
}

// The stem through the halo engine: space-to-depth of x and the filter into
// the workspace, then a 4x4 stride-1 convolution over 16 channels with 32-byte
// pixel rows (layouts at stem_s2d_width).  y is N x P x Q x 64.
int run_stem_s2d(const Shape& s, int ws, const uint16_t* x, const uint16_t* w, uint16_t* y, void* work,
                 int* status, int sms, cudaStream_t st, void* stats, bool f32) {
  const long long N = s.N, P = s.P, Q = s.Q, Hs = P + 3, Wsd = Q + 3;
  uint16_t* xs = static_cast<uint16_t*>(work);
  uint16_t* wsd = xs + stem_s2d_bytes(s) / 2;
  if (launch_stem_s2d(x, w, xs, wsd, (int)N, (int)s.H, (int)s.W, (int)Hs, (int)Wsd, (int)s.K, st) != cudaSuccess)
    return PF16_ERR_CUDA;
  GemmParams p = base_params(status);
  set_stats(p, stats, 64);
  p.d_f32 = f32 ? 1 : 0;
  CUtensorMap ma, mb, mc;
  const int rows = kBM / ws;
  cuuint64_t dims[4] = {16, (cuuint64_t)Wsd, (cuuint64_t)Hs, (cuuint64_t)N};
  cuuint64_t strides[3] = {32, (cuuint64_t)(Wsd * 32), (cuuint64_t)(Hs * Wsd * 32)};
  cuuint32_t box[4] = {16, (cuuint32_t)ws, (cuuint32_t)(rows + 3), 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  if (g_encode_tiled(&ma, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, xs, dims, strides, box, es,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_32B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return PF16_ERR_CUDA;
  if (!map_2d(&mb, wsd, 256, 64, 256, 16, 64, CU_TENSOR_MAP_SWIZZLE_32B)) return PF16_ERR_CUDA;
  if (!map_3d(&mc, y, 64, Q, N * P, 128, Q * 128, 64, 32, 1)) return PF16_ERR_CUDA;
  p.ntaps = 16;
  for (int t = 0; t < 16; ++t) {
    p.tap_dr[t] = (int8_t)(t / 4);
    p.tap_ds[t] = (int8_t)(t % 4);
    p.tap_w[t] = (int8_t)t;
  }
  p.b_mode = LD_TILED_K;
  p.b_lbo = 16;
  p.b_sbo = 256;  // 8 rows of 32 bytes
  p.b_kstep = 32;
  p.idesc = idesc_f16(kBM, 64, false, false, f32);
  p.halo_ws = ws;
  p.halo_h = (int)P;
  p.halo_w = (int)Q;
  p.halo_cb = 32;
  p.halo_box_rows = rows + 3;
  p.halo_row0 = 0;
  p.halo_col0 = 0;
  p.N = 64;
  p.n_tiles = 1;
  p.m_tiles = (int)(N * P * ws / kBM);
  int grid = p.m_tiles < sms ? p.m_tiles : sms;
  if (stats && grid > kBnStatSlots) grid = kBnStatSlots;
  return launch_gemm_halo(ma, mb, mc, p, grid, st) == cudaSuccess ? PF16_OK : PF16_ERR_CUDA;
}

// BatchNorm in the operand path: validate `bn` for an input of C channels
// and point the GEMM's transform at it (xf_operand 1: A, 2: B).
static int set_bn_operand(GemmParams& p, const pf16_bn_operand* bn, long long C, long long rows, int operand,
                          bool allow_mask) {
  if (!bn->mean || !bn->invstd || !bn->gamma || !bn->beta) return PF16_ERR_NULL;
  if (!aligned16(bn->mean) || !aligned16(bn->invstd) || !aligned16(bn->gamma) || !aligned16(bn->beta))
    return PF16_ERR_ALIGN;
  if (bn->flags & ~(uint32_t)PF16_BN_RELU) return PF16_ERR_ARG;
  if (bn->relu_mask && (!allow_mask || !(bn->flags & PF16_BN_RELU))) return PF16_ERR_ARG;
  if (C % 8 != 0) return PF16_ERR_UNSUPPORTED;
  p.xf_operand = operand;
  p.xf_relu = (bn->flags & PF16_BN_RELU) ? 1 : 0;
  p.xf_scale = bn->post_scale;
  p.xf_C = (int)C;
  p.xf_rows = rows;
  p.xf_mean = bn->mean;
  p.xf_invstd = bn->invstd;
  p.xf_gamma = bn->gamma;
  p.xf_beta = bn->beta;
  p.xf_mask = bn->relu_mask;
  return PF16_OK;
}

static int conv_fwd_impl(const pf16_conv_desc* d, const uint16_t* x, const uint16_t* w, uint16_t* y,
                         void* ws, size_t ws_bytes, uint32_t flags, void* stats, size_t stats_bytes,
                         void* stream, const pf16_bn_operand* bn = nullptr) {
  Shape s;
  int rc = conv_shape(d, &s);
  if (rc != PF16_OK) return rc;
  if ((rc = check_common(x, w, y)) != PF16_OK) return rc;
  const bool dense = s.kind == KIND_GENERIC && s.R == 1 && s.S == 1 && s.st == 1 && s.pad == 0;
  if (bn && (!dense || flags != 0)) return PF16_ERR_UNSUPPORTED;
  if (flags & ~(PF16_ACCUMULATE | PF16_F32_ACCUM)) return PF16_ERR_ARG;
  const bool f32 = (flags & PF16_F32_ACCUM) != 0;
  if (stats) {
    if (flags != 0) return PF16_ERR_ARG;  // statistics of a plain (non-accumulating) output only
    if (s.K % 64 != 0) return PF16_ERR_UNSUPPORTED;
    if (!aligned16(stats)) return PF16_ERR_ALIGN;
    if (stats_bytes < bnstat_bytes(s.K)) return PF16_ERR_WORKSPACE;
  }
  const size_t need = ws_fwd(s);
  if (need && (!ws || ws_bytes < need)) return PF16_ERR_WORKSPACE;
  if (need && !aligned16(ws)) return PF16_ERR_ALIGN;
  if (!driver_fns()) return PF16_ERR_CUDA;
  int* status;
  int sms;
  if ((rc = device_consts(&status, &sms)) != PF16_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);

  GemmParams p = base_params(status);
  p.d_f32 = f32 ? 1 : 0;
  CUtensorMap ma, mb;
  p.M = (int)(s.N * s.P * s.Q);
  p.N = (int)s.K;
  p.out = y;
  p.ldo = s.K;
  p.out_mode = (flags & PF16_ACCUMULATE) ? OUT_ACCUM : OUT_STORE;
  if (bn && (rc = set_bn_operand(p, bn, s.C, (long long)p.M, 1, true)) != PF16_OK) return rc;
  if (const int ws = bn ? 0 : halo_width(s, (flags & PF16_ACCUMULATE) != 0))
    return run_halo(s, ws, false, x, w, y, status, sms, st, f32, stats);
  if (!bn) {
    const WidePlan wp = halo_wide_plan(s, s.C, s.K, (flags & PF16_ACCUMULATE) != 0);
    if (wp.ipr) return run_halo_wide(s, wp, x, w, y, status, sms, st, f32, stats);
  }
  if (const int ws_s2d = stem_s2d_width(s, (flags & PF16_ACCUMULATE) != 0))
    return run_stem_s2d(s, ws_s2d, x, w, y, ws, status, sms, st, stats, f32);
  set_stats(p, stats, s.K);
  const int BN = pick_bn_out(s.K);
  p.a_mode = LD_TILED_K;
  p.b_mode = LD_TILED_K;
  set_kmajor(p, true, true);
  if (s.kind == KIND_STEM) {
    const long long kc = stem_kcol(s);
    uint16_t* col = static_cast<uint16_t*>(ws);
    uint16_t* wpad = col + round_up((size_t)(p.M * kc * 2), 256) / 2;
    if (launch_stem_im2col(x, col, (int)s.N, (int)s.H, (int)s.W, (int)s.P, (int)s.Q, (int)s.R,
                           (int)s.S, (int)s.C, (int)s.st, (int)s.pad, (int)kc, st) != cudaSuccess)
      return PF16_ERR_CUDA;
    if (launch_pad_rows(w, wpad, (int)s.K, (int)(s.R * s.S * s.C), (int)kc, st) != cudaSuccess)
      return PF16_ERR_CUDA;
    if (!map_2d(&ma, col, kc, p.M, kc, 64, kBM) || !map_2d(&mb, wpad, kc, s.K, kc, 64, BN))
      return PF16_ERR_CUDA;
    p.num_kb = cdiv(kc, kBK);
  } else {
    if (dense) {
      if (!map_2d(&ma, x, s.C, s.N * s.H * s.W, s.C, 64, kBM)) return PF16_ERR_CUDA;
    } else {
      p.a_mode = LD_IM2COL_K;
      p.ga = PixGrid{(int)s.P, (int)s.Q, (int)s.st, (int)-s.pad, (int)-s.pad};
      if (!map_im2col(&ma, x, (int)s.N, (int)s.H, (int)s.W, (int)s.C, (int)-s.pad, (int)-s.pad,
                      (int)s.P, (int)s.Q, (int)s.st, kBM))
        return PF16_ERR_CUDA;
      p.ntaps = (int)(s.R * s.S);
      for (int r = 0; r < s.R; ++r)
        for (int c = 0; c < s.S; ++c) {
          p.tap_dr[r * s.S + c] = (int8_t)r;
          p.tap_ds[r * s.S + c] = (int8_t)c;
          p.tap_w[r * s.S + c] = (int8_t)(r * s.S + c);
        }
      p.a_cpt = (int)(s.C / 64);
    }
    if (!map_2d(&mb, w, s.R * s.S * s.C, s.K, s.R * s.S * s.C, 64, BN)) return PF16_ERR_CUDA;
    p.num_kb = (int)(s.R * s.S * s.C / 64);
  }
  return run(BN, ma, mb, p, sms, st);
}

int pf16_conv_fwd(const pf16_conv_desc* d, const uint16_t* x, const uint16_t* w, uint16_t* y,
                  void* ws, size_t ws_bytes, uint32_t flags, void* stream) {
  return conv_fwd_impl(d, x, w, y, ws, ws_bytes, flags, nullptr, 0, stream);
}

size_t pf16_conv_bnstats_size(const pf16_conv_desc* d) {
  Shape s;
  if (conv_shape(d, &s) != PF16_OK || s.K % 64 != 0) return 0;
  return bnstat_bytes(s.K);
}

int pf16_conv_fwd_bnstats(const pf16_conv_desc* d, const uint16_t* x, const uint16_t* w, uint16_t* y,
                          void* ws, size_t ws_bytes, void* stats, size_t stats_bytes, void* stream) {
  if (!stats) return PF16_ERR_NULL;
  return conv_fwd_impl(d, x, w, y, ws, ws_bytes, 0, stats, stats_bytes, stream);
}

int pf16_conv_fwd_bnin(const pf16_conv_desc* d, const uint16_t* x, const pf16_bn_operand* bn, const uint16_t* w,
                       uint16_t* y, void* stats, size_t stats_bytes, void* stream) {
  if (!bn) return PF16_ERR_NULL;
  return conv_fwd_impl(d, x, w, y, nullptr, 0, 0, stats, stats_bytes, stream, bn);
}

static int conv_dgrad_impl(const pf16_conv_desc* d, const uint16_t* dy, const uint16_t* w, uint16_t* dx,
                           uint32_t flags, void* stats, size_t stats_bytes, const pf16_bn_source* bn,
                           void* stream, const uint16_t* add = nullptr, const uint8_t* add_mask = nullptr) {
  Shape s;
  int rc = conv_shape(d, &s);
  if (rc != PF16_OK) return rc;
  if (s.kind == KIND_STEM) return PF16_ERR_UNSUPPORTED;
  if ((rc = check_common(dy, w, dx)) != PF16_OK) return rc;
  if (flags & ~(PF16_ACCUMULATE | PF16_F32_ACCUM)) return PF16_ERR_ARG;
  const bool f32 = (flags & PF16_F32_ACCUM) != 0;
  if (stats) {
    // statistics of a plain output whose rows are pixels in order (stride 1)
    if (flags != 0) return PF16_ERR_ARG;
    if (!bn->x || !bn->mean || !bn->invstd) return PF16_ERR_NULL;
    if (!aligned16(stats) || !aligned16(bn->x) || !aligned16(bn->mean) || !aligned16(bn->invstd) ||
        (reinterpret_cast<uintptr_t>(bn->relu_mask) & 7u) != 0)
      return PF16_ERR_ALIGN;
    if (s.C % 64 != 0 || (s.st != 1 && !phases_one_launch(s))) return PF16_ERR_UNSUPPORTED;
    if (stats_bytes < bnstat_bytes(s.C)) return PF16_ERR_WORKSPACE;
  }
  if (add) {
    // the masked addend: a plain 1x1 data gradient (one GEMM, rows in pixel order)
    if (!stats) return PF16_ERR_ARG;
    if (s.R != 1 || s.S != 1 || s.pad != 0) return PF16_ERR_UNSUPPORTED;
    if (!aligned16(add) || (reinterpret_cast<uintptr_t>(add_mask) & 7u) != 0) return PF16_ERR_ALIGN;
    const size_t bytes = (size_t)(s.N * s.H * s.W * s.C) * 2;
    const uintptr_t a0 = reinterpret_cast<uintptr_t>(add), d0 = reinterpret_cast<uintptr_t>(dx);
    if (a0 < d0 + bytes && d0 < a0 + bytes) return PF16_ERR_ARG;  // read through the read-only path
  }
  if (!driver_fns()) return PF16_ERR_CUDA;
  int* status;
  int sms;
  if ((rc = device_consts(&status, &sms)) != PF16_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const bool accum = (flags & PF16_ACCUMULATE) != 0;
  if (const int ws = halo_width(s, accum))
    return run_halo(s, ws, true, dy, w, dx, status, sms, st, f32, stats, stats ? bn : nullptr);
  // with an addend the TMA-fed epilogue leaves 256-wide tiles two pipeline
  // stages; reductions of 4+ K-blocks keep three with 128-wide tiles
  const int BN = (add && s.K >= 4 * kBK) ? std::min(pick_bn_out(s.C), 128) : pick_bn_out(s.C);
  const size_t dx_elems = (size_t)(s.N * s.H * s.W * s.C);

  if (s.R == 1 && s.S == 1 && s.pad == 0) {
    // 1x1: dx[n, st*p, st*q, :] = dy[n,p,q,:] . w ; other positions receive nothing
    GemmParams p = base_params(status);
    p.d_f32 = f32 ? 1 : 0;
    set_stats(p, stats, s.C);
    if (stats) set_bwd_stats(p, bn);
    p.add_src = add;
    p.add_mask = add ? add_mask : nullptr;
    CUtensorMap ma, mb;
    p.M = (int)(s.N * s.P * s.Q);
    p.N = (int)s.C;
    p.a_mode = LD_TILED_K;
    p.b_mode = LD_TILED_MN;
    set_kmajor(p, true, false);
    set_mnmajor(p, false, true);
    if (!map_2d(&ma, dy, s.K, s.N * s.P * s.Q, s.K, 64, kBM) ||
        !map_2d(&mb, w, s.C, s.K, s.C, 64, 64))
      return PF16_ERR_CUDA;
    p.num_kb = cdiv(s.K, kBK);
    p.out = dx;
    p.ldo = s.C;
    p.out_mode = accum ? OUT_ACCUM : OUT_STORE;
    if (s.st != 1) {
      if (!accum && launch_fill_zero(dx, dx_elems, st) != cudaSuccess) return PF16_ERR_CUDA;
      p.remap = 1;
      p.rm_gh = (int)s.P;
      p.rm_gw = (int)s.Q;
      p.rm_H = (int)s.H;
      p.rm_W = (int)s.W;
      p.rm_step = (int)s.st;
    }
    return run(BN, ma, mb, p, sms, st);
  }

  // R x S filters: one implicit GEMM per stride phase (ph, pw); positions no
  // phase reaches are zero-filled first (unless accumulating).
  bool any_empty = false;
  for (int ph = 0; ph < s.st; ++ph)
    for (int pw = 0; pw < s.st; ++pw) any_empty |= make_phase(s, ph, pw).empty();
  if (phases_one_launch(s)) return run_dgrad_phases(s, dy, w, dx, status, sms, st, f32, accum, BN, stats, bn);
  if (any_empty && !accum && launch_fill_zero(dx, dx_elems, st) != cudaSuccess)
    return PF16_ERR_CUDA;
  for (int ph = 0; ph < s.st; ++ph)
    for (int pw = 0; pw < s.st; ++pw) {
      const Phase f = make_phase(s, ph, pw);
      if (f.empty()) continue;
      const int gh = f.gh, gw = f.gw, nr = f.nr, ns = f.ns;
      const int *ar = f.ar, *bs = f.bs, *rr = f.rr, *ss = f.ss;
      const int amin = *std::min_element(ar, ar + nr), bmin = *std::min_element(bs, bs + ns);
      GemmParams p = base_params(status);
      p.d_f32 = f32 ? 1 : 0;
      set_stats(p, stats, s.C);  // stride 1 only: one phase, rows in pixel order
      if (stats) set_bwd_stats(p, bn);
      CUtensorMap ma, mb;
      p.M = (int)(s.N * gh * gw);
      p.N = (int)s.C;
      p.a_mode = LD_IM2COL_K;
      p.b_mode = LD_TAP3D_MN;
      set_kmajor(p, true, false);
      set_mnmajor(p, false, true);
      p.ga = PixGrid{gh, gw, 1, amin, bmin};
      if (!map_im2col(&ma, dy, (int)s.N, (int)s.P, (int)s.Q, (int)s.K, amin, bmin, gh, gw, 1, kBM))
        return PF16_ERR_CUDA;
      if (!map_3d(&mb, w, s.C, s.R * s.S, s.K, s.C * 2, s.R * s.S * s.C * 2, 64, 1, 64))
        return PF16_ERR_CUDA;
      p.ntaps = nr * ns;
      for (int i = 0; i < nr; ++i)
        for (int j = 0; j < ns; ++j) {
          p.tap_dr[i * ns + j] = (int8_t)(ar[i] - amin);
          p.tap_ds[i * ns + j] = (int8_t)(bs[j] - bmin);
          p.tap_w[i * ns + j] = (int8_t)(rr[i] * s.S + ss[j]);
        }
      p.a_cpt = p.b_cpt = (int)(s.K / 64);
      p.num_kb = p.ntaps * p.a_cpt;
      p.out = dx;
      p.ldo = s.C;
      p.out_mode = accum ? OUT_ACCUM : OUT_STORE;
      p.remap = (s.st != 1) ? 1 : 0;
      p.rm_gh = gh;
      p.rm_gw = gw;
      p.rm_H = (int)s.H;
      p.rm_W = (int)s.W;
      p.rm_step = (int)s.st;
      p.rm_ph = ph;
      p.rm_pw = pw;
      if ((rc = run(BN, ma, mb, p, sms, st)) != PF16_OK) return rc;
    }
  return PF16_OK;
}

int pf16_conv_dgrad(const pf16_conv_desc* d, const uint16_t* dy, const uint16_t* w, uint16_t* dx,
                    void* ws, size_t ws_bytes, uint32_t flags, void* stream) {
  (void)ws;
  (void)ws_bytes;
  return conv_dgrad_impl(d, dy, w, dx, flags, nullptr, 0, nullptr, stream);
}

size_t pf16_conv_dgrad_bnstats_size(const pf16_conv_desc* d) {
  Shape s;
  if (conv_shape(d, &s) != PF16_OK || s.kind == KIND_STEM || s.C % 64 != 0) return 0;
  if (s.st != 1 && !phases_one_launch(s)) return 0;
  return bnstat_bytes(s.C);
}

int pf16_conv_dgrad_bnstats(const pf16_conv_desc* d, const uint16_t* dy, const uint16_t* w, uint16_t* dx,
                            void* ws, size_t ws_bytes, const pf16_bn_source* bn, void* stats,
                            size_t stats_bytes, void* stream) {
  (void)ws;
  (void)ws_bytes;
  if (!bn || !stats) return PF16_ERR_NULL;
  return conv_dgrad_impl(d, dy, w, dx, 0, stats, stats_bytes, bn, stream);
}

int pf16_conv_dgrad_bnstats_add(const pf16_conv_desc* d, const uint16_t* dy, const uint16_t* w, uint16_t* dx,
                                void* ws, size_t ws_bytes, const pf16_bn_source* bn, const uint16_t* add,
                                const uint8_t* add_mask, void* stats, size_t stats_bytes, void* stream) {
  (void)ws;
  (void)ws_bytes;
  if (!bn || !stats || !add) return PF16_ERR_NULL;
  return conv_dgrad_impl(d, dy, w, dx, 0, stats, stats_bytes, bn, stream, add, add_mask);
}

// The stem's weight gradient through k_stem_wgrad (layouts at stem_wgrad_plan).
static int run_stem_wgrad(const Shape& s, const StemWgradPlan& sw, const uint16_t* x, const uint16_t* dy,
                          uint16_t* dw, void* work, int* status, int sms, cudaStream_t st, bool f32) {
  const long long N = s.N, P = s.P, Q = s.Q, Hs = P + 3, Wsd = Q + 3;
  uint16_t* xs = static_cast<uint16_t*>(work);
  uint16_t* parts = xs + stem_s2d_bytes(s) / 2;
  uint16_t* dws = parts + stem_wgrad_parts_bytes(sw) / 2;
  if (launch_stem_s2d(x, nullptr, xs, nullptr, (int)N, (int)s.H, (int)s.W, (int)Hs, (int)Wsd, 0, st) !=
      cudaSuccess)
    return PF16_ERR_CUDA;
  CUtensorMap mdy, mxs;
  cuuint32_t es[4] = {1, 1, 1, 1};
  {
    cuuint64_t dims[4] = {64, (cuuint64_t)Q, (cuuint64_t)P, (cuuint64_t)N};
    cuuint64_t strides[3] = {128, (cuuint64_t)(Q * 128), (cuuint64_t)(P * Q * 128)};
    cuuint32_t box[4] = {64, 128, 2, 1};
    if (g_encode_tiled(&mdy, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<uint16_t*>(dy), dims, strides, box, es,
                       CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                       CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return PF16_ERR_CUDA;
  }
  {
    cuuint64_t dims[4] = {16, (cuuint64_t)Wsd, (cuuint64_t)Hs, (cuuint64_t)N};
    cuuint64_t strides[3] = {32, (cuuint64_t)(Wsd * 32), (cuuint64_t)(Hs * Wsd * 32)};
    cuuint32_t box[4] = {16, 128, 4, 1};
    if (g_encode_tiled(&mxs, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, xs, dims, strides, box, es,
                       CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_32B,
                       CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return PF16_ERR_CUDA;
  }
  GemmParams p = base_params(status);
  p.d_f32 = f32 ? 1 : 0;
  p.idesc = idesc_f16(kBM, 64, true, true, f32);
  p.halo_ws = 128;
  p.halo_h = (int)P;
  p.halo_w = (int)Q;
  p.num_kb = (int)sw.rows;
  p.kb_per_split = sw.per_chunk;
  p.m_tiles = sw.chunks;
  p.out = parts;
  const int grid = sw.chunks < sms ? sw.chunks : sms;
  if (launch_stem_wgrad(mdy, mxs, p, grid, st) != cudaSuccess) return PF16_ERR_CUDA;
  if (launch_splitk_reduce(parts, sw.chunks, 128, 128, dws, 128, 128, st) != cudaSuccess) return PF16_ERR_CUDA;
  if (launch_stem_wgrad_scatter(dws, dw, (int)s.K, st) != cudaSuccess) return PF16_ERR_CUDA;
  return PF16_OK;
}

// The 3x3, 64 -> 64 weight gradient through k_wgrad3x3_halo (layouts at
// wgrad3_plan), then the split-K tree straight into dw.
static int run_wgrad3x3(const Shape& s, const Wgrad3Plan& w3, const uint16_t* x, const uint16_t* dy, uint16_t* dw,
                        void* work, int* status, int sms, cudaStream_t st, bool f32) {
  const long long N = s.N, H = s.H, W = s.W, P = s.P, Q = s.Q;
  uint16_t* parts = static_cast<uint16_t*>(work);
  CUtensorMap mdy, mx;
  cuuint32_t es[4] = {1, 1, 1, 1};
  {
    cuuint64_t dims[4] = {64, (cuuint64_t)Q, (cuuint64_t)P, (cuuint64_t)N};
    cuuint64_t strides[3] = {128, (cuuint64_t)(Q * 128), (cuuint64_t)(P * Q * 128)};
    cuuint32_t box[4] = {64, 64, 3, 1};
    if (g_encode_tiled(&mdy, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<uint16_t*>(dy), dims, strides, box, es,
                       CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                       CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return PF16_ERR_CUDA;
  }
  {
    cuuint64_t dims[4] = {64, (cuuint64_t)W, (cuuint64_t)H, (cuuint64_t)N};
    cuuint64_t strides[3] = {128, (cuuint64_t)(W * 128), (cuuint64_t)(H * W * 128)};
    cuuint32_t box[4] = {64, 64, 4, 1};
    if (g_encode_tiled(&mx, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<uint16_t*>(x), dims, strides, box, es,
                       CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                       CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return PF16_ERR_CUDA;
  }
  GemmParams p = base_params(status);
  p.d_f32 = f32 ? 1 : 0;
  p.idesc = idesc_f16(kBM, 192, true, true, f32);
  p.halo_ws = 64;
  p.halo_h = (int)P;
  p.halo_w = (int)Q;
  p.num_kb = (int)w3.units;
  p.kb_per_split = w3.per_chunk;
  p.m_tiles = w3.chunks;
  p.out = parts;
  const int grid = w3.chunks < sms ? w3.chunks : sms;
  if (launch_wgrad3x3_halo(mdy, mx, p, grid, st) != cudaSuccess) return PF16_ERR_CUDA;
  if (launch_splitk_reduce(parts, w3.chunks, 64, 576, dw, 576, 576, st) != cudaSuccess) return PF16_ERR_CUDA;
  return PF16_OK;
}

// The 3x3 stride-1 weight gradient with K % 128 == 0 through
// k_wgrad3x3_wide (layouts at wide_wgrad_plan), then the split-K tree
// straight into dw.
static int run_wgrad3x3_wide(const Shape& s, const WideWgradPlan& ww, const uint16_t* x, const uint16_t* dy,
                             uint16_t* dw, void* work, int* status, int sms, cudaStream_t st, bool f32) {
  const long long N = s.N, H = s.H, W = s.W, C = s.C, K = s.K;
  uint16_t* parts = static_cast<uint16_t*>(work);
  CUtensorMap mdy, mx;
  cuuint32_t es[4] = {1, 1, 1, 1};
  cuuint32_t box[4] = {64, (cuuint32_t)ww.wi, (cuuint32_t)ww.nb, 1};
  // both maps (c, w, n, h) over an NHWC tensor
  for (int m = 0; m < 2; ++m) {
    const long long ch = m == 0 ? K : C;
    const cuuint64_t pix = (cuuint64_t)ch * 2, row = (cuuint64_t)W * pix, img = (cuuint64_t)H * row;
    cuuint64_t dims[4] = {(cuuint64_t)ch, (cuuint64_t)W, (cuuint64_t)N, (cuuint64_t)H};
    cuuint64_t strides[3] = {pix, img, row};
    void* base = const_cast<uint16_t*>(m == 0 ? dy : x);
    if (g_encode_tiled(m == 0 ? &mdy : &mx, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, base, dims, strides, box, es,
                       CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                       CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return PF16_ERR_CUDA;
  }
  GemmParams p = base_params(status);
  p.d_f32 = f32 ? 1 : 0;
  p.idesc = idesc_f16(kBM, 192, true, true, f32);
  p.M = (int)K;
  p.halo_chunks = (int)(C / 64);
  p.halo_wi = ww.wi;
  p.halo_ipr = ww.nb;
  p.halo_w = (int)W;
  p.halo_h = (int)H;
  p.num_kb = (int)ww.tiles;
  p.kb_per_split = ww.per_chunk;
  p.splits = ww.chunks;
  p.m_tiles = ww.chunks * ww.types;
  p.out = parts;
  p.ldo = 9 * C;
  const int grid = p.m_tiles < sms ? p.m_tiles : sms;
  if (launch_wgrad3x3_wide(mdy, mx, p, grid, st) != cudaSuccess) return PF16_ERR_CUDA;
  if (launch_splitk_reduce(parts, ww.chunks, K, (int)(9 * C), dw, 9 * C, (int)(9 * C), st) != cudaSuccess)
    return PF16_ERR_CUDA;
  return PF16_OK;
}

static int conv_wgrad_impl(const pf16_conv_desc* d, const uint16_t* x, const uint16_t* dy, uint16_t* dw,
                           void* ws, size_t ws_bytes, uint32_t flags, void* stream,
                           const pf16_bn_operand* bn = nullptr) {
  Shape s;
  int rc = conv_shape(d, &s);
  if (rc != PF16_OK) return rc;
  if ((rc = check_common(x, dy, dw)) != PF16_OK) return rc;
  if (flags & ~PF16_F32_ACCUM) return PF16_ERR_ARG;
  const bool dense = s.kind == KIND_GENERIC && s.R == 1 && s.S == 1 && s.st == 1 && s.pad == 0;
  if (bn && (!dense || flags != 0)) return PF16_ERR_UNSUPPORTED;
  const bool f32 = (flags & PF16_F32_ACCUM) != 0;
  int* status;
  int sms;
  if ((rc = device_consts(&status, &sms)) != PF16_OK) return rc;
  const size_t need = ws_wgrad(s);
  if (need && (!ws || ws_bytes < need)) return PF16_ERR_WORKSPACE;
  if (need && !aligned16(ws)) return PF16_ERR_ALIGN;
  if (!driver_fns()) return PF16_ERR_CUDA;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const StemWgradPlan sw = stem_wgrad_plan(s);
  if (sw.ok) return run_stem_wgrad(s, sw, x, dy, dw, ws, status, sms, st, f32);
  const Wgrad3Plan w3 = wgrad3_plan(s);
  if (w3.ok) return run_wgrad3x3(s, w3, x, dy, dw, ws, status, sms, st, f32);
  const WideWgradPlan ww = wide_wgrad_plan(s);
  if (ww.ok) return run_wgrad3x3_wide(s, ww, x, dy, dw, ws, status, sms, st, f32);
  const WgradSplit wsp = wgrad_split(s);

  GemmParams p = base_params(status);
  p.d_f32 = f32 ? 1 : 0;
  CUtensorMap ma, mb;
  const long long pixels = s.N * s.P * s.Q;
  p.M = (int)s.K;
  p.N = (int)wsp.ncols;
  p.num_kb = wsp.num_kb;
  p.splits = wsp.splits;
  p.kb_per_split = wsp.kb_per_split;
  p.a_mode = LD_TILED_MN;
  set_mnmajor(p, true, true);
  if (!map_2d(&ma, dy, s.K, pixels, s.K, 64, 64)) return PF16_ERR_CUDA;
  // stem: [patch matrix][partials]; other layers: [partials]
  uint16_t* parts = static_cast<uint16_t*>(ws);
  const bool partial = wsp.splits > 1 || s.kind == KIND_STEM;
  if (s.kind == KIND_STEM) {
    uint16_t* col = static_cast<uint16_t*>(ws);
    parts = col + round_up((size_t)(pixels * wsp.ncols * 2), 256) / 2;
    if (launch_stem_im2col(x, col, (int)s.N, (int)s.H, (int)s.W, (int)s.P, (int)s.Q, (int)s.R,
                           (int)s.S, (int)s.C, (int)s.st, (int)s.pad, (int)wsp.ncols,
                           st) != cudaSuccess)
      return PF16_ERR_CUDA;
    p.b_mode = LD_TILED_MN;
    if (!map_2d(&mb, col, wsp.ncols, pixels, wsp.ncols, 64, 64)) return PF16_ERR_CUDA;
  } else if (s.R == 1 && s.S == 1 && s.st == 1 && s.pad == 0) {
    p.b_mode = LD_TILED_MN;
    if (!map_2d(&mb, x, s.C, pixels, s.C, 64, 64)) return PF16_ERR_CUDA;
    if (bn && (rc = set_bn_operand(p, bn, s.C, pixels, 2, false)) != PF16_OK) return rc;
  } else {
    p.b_mode = LD_IM2COL_MN;
    p.gb = PixGrid{(int)s.P, (int)s.Q, (int)s.st, (int)-s.pad, (int)-s.pad};
    if (!map_im2col(&mb, x, (int)s.N, (int)s.H, (int)s.W, (int)s.C, (int)-s.pad, (int)-s.pad,
                    (int)s.P, (int)s.Q, (int)s.st, 64))
      return PF16_ERR_CUDA;
    p.ntaps = (int)(s.R * s.S);
    for (int r = 0; r < s.R; ++r)
      for (int c = 0; c < s.S; ++c) {
        p.tap_dr[r * s.S + c] = (int8_t)r;
        p.tap_ds[r * s.S + c] = (int8_t)c;
      }
    p.b_cin = (int)s.C;
    p.b_oob_c = (int)round_up((size_t)s.C, 64);
  }
  if (partial) {
    p.out = parts;
    p.ldo = wsp.ncols;
    p.out_mode = OUT_PARTIAL;
  } else {
    p.out = dw;
    p.ldo = wsp.ncols;
    p.out_mode = OUT_STORE;
  }
  if ((rc = run(wsp.bn, ma, mb, p, sms, st)) != PF16_OK) return rc;
  if (partial) {
    const long long rsc = s.R * s.S * s.C;
    if (launch_splitk_reduce(parts, wsp.splits, s.K, (int)wsp.ncols, dw, rsc, (int)rsc, st) !=
        cudaSuccess)
      return PF16_ERR_CUDA;
  }
  return PF16_OK;
}

int pf16_conv_wgrad(const pf16_conv_desc* d, const uint16_t* x, const uint16_t* dy, uint16_t* dw,
                    void* ws, size_t ws_bytes, uint32_t flags, void* stream) {
  return conv_wgrad_impl(d, x, dy, dw, ws, ws_bytes, flags, stream);
}

int pf16_conv_wgrad_bnin(const pf16_conv_desc* d, const uint16_t* x, const pf16_bn_operand* bn, const uint16_t* dy,
                         uint16_t* dw, void* ws, size_t ws_bytes, void* stream) {
  if (!bn) return PF16_ERR_NULL;
  return conv_wgrad_impl(d, x, dy, dw, ws, ws_bytes, 0, stream, bn);
}

int pf16_sgd_update(uint16_t* w, uint16_t* v, const uint16_t* g, size_t n, uint16_t lr,
                    uint16_t momentum, uint16_t wd, uint32_t flags, void* stream) {
  if (flags != 0) return PF16_ERR_ARG;
  if (n == 0) return PF16_OK;
  if (!w || !v || !g) return PF16_ERR_NULL;
  if (!aligned16(w) || !aligned16(v) || !aligned16(g)) return PF16_ERR_ALIGN;
  return launch_sgd(w, v, g, n, lr, momentum, wd, static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? PF16_OK
             : PF16_ERR_CUDA;
}

int pf16_allreduce_combine(const uint16_t* planes, int32_t world, size_t n, size_t plane_stride,
                           uint16_t scale, uint16_t* out, void* stream) {
  if (world < 1 || world > 1024 || n % 8 != 0 || plane_stride % 8 != 0 || plane_stride < n)
    return PF16_ERR_SHAPE;
  if ((size_t)world * plane_stride > ((size_t)1 << 40)) return PF16_ERR_SHAPE;
  if (n == 0) return PF16_OK;
  if (!planes || !out) return PF16_ERR_NULL;
  if (!aligned16(planes) || !aligned16(out)) return PF16_ERR_ALIGN;
  // out is plane 0 or lies clear of every plane
  const uintptr_t o = reinterpret_cast<uintptr_t>(out), b = reinterpret_cast<uintptr_t>(planes);
  const uintptr_t e = b + ((size_t)(world - 1) * plane_stride + n) * 2;
  if (o != b && o + n * 2 > b && o < e) return PF16_ERR_SHAPE;
  return launch_dp_combine(planes, world, n, plane_stride, scale, out, static_cast<cudaStream_t>(stream)) ==
                 cudaSuccess
             ? PF16_OK
             : PF16_ERR_CUDA;
}

static int bn_validate(const pf16_bn_desc* d, BnLaunch* b) {
  if (!d) return PF16_ERR_NULL;
  if (d->n <= 0 || d->h <= 0 || d->w <= 0 || d->c <= 0) return PF16_ERR_SHAPE;
  if (d->c % 8 != 0 || d->c > 2048) return PF16_ERR_UNSUPPORTED;
  if (d->flags & ~(uint32_t)(PF16_BN_RELU | PF16_BN_RESIDUAL | PF16_BN_SWAP)) return PF16_ERR_ARG;
  if ((d->flags & PF16_BN_SWAP) && !(d->flags & PF16_BN_RESIDUAL)) return PF16_ERR_ARG;
  const long long R = (long long)d->n * d->h * d->w;
  if (R * d->c > (1ll << 34) || R > (1ll << 31) - 1) return PF16_ERR_SHAPE;
  bn_plan((int)R, d->c, b);
  b->eps = d->eps;
  b->post_scale = d->post_scale;
  b->relu = (d->flags & PF16_BN_RELU) ? 1 : 0;
  b->residual = (d->flags & PF16_BN_RESIDUAL) ? 1 : 0;
  b->swap = (d->flags & PF16_BN_SWAP) ? 1 : 0;
  return PF16_OK;
}

size_t pf16_bn_workspace_size(const pf16_bn_desc* d) {
  BnLaunch b;
  if (bn_validate(d, &b) != PF16_OK) return 0;
  return bn_ws_bytes(b);
}

int pf16_bn_fwd_bwd(const pf16_bn_desc* d, int phase, const pf16_bn_tensors* t, void* ws,
                    size_t ws_bytes, void* stream) {
  BnLaunch b;
  int rc = bn_validate(d, &b);
  if (rc != PF16_OK) return rc;
  if (!t) return PF16_ERR_NULL;
  if (phase != 0 && phase != 1) return PF16_ERR_ARG;
  if (!ws) return PF16_ERR_WORKSPACE;
  if (ws_bytes < bn_ws_bytes(b)) return PF16_ERR_WORKSPACE;
  if (!aligned16(ws)) return PF16_ERR_ALIGN;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int sms = 0;
  if (phase == 0) {
    // y == NULL: the statistics only (mean, invstd), for a consumer that
    // applies the BatchNorm in its operand path
    const void* req[] = {t->x, t->mean, t->invstd};
    for (const void* p : req) {
      if (!p) return PF16_ERR_NULL;
      if (!aligned16(p)) return PF16_ERR_ALIGN;
    }
    if (t->y) {
      const void* req2[] = {t->gamma, t->beta, t->y};
      for (const void* p : req2) {
        if (!p) return PF16_ERR_NULL;
        if (!aligned16(p)) return PF16_ERR_ALIGN;
      }
      if (b.residual && !t->residual) return PF16_ERR_NULL;
      if (b.residual && !aligned16(t->residual)) return PF16_ERR_ALIGN;
    } else if (t->relu_mask) {
      return PF16_ERR_ARG;  // the decisions come from the apply
    }
    if (device_consts(&b.status, &sms) != PF16_OK) return PF16_ERR_CUDA;
    if (t->conv_stats) {
      if (!aligned16(t->conv_stats)) return PF16_ERR_ALIGN;
      return launch_bn_fwd_given_stats(b, static_cast<const uint8_t*>(t->conv_stats), t->x, t->gamma,
                                       t->beta, b.residual ? t->residual : nullptr, t->y, t->relu_mask,
                                       t->mean, t->invstd, st) == cudaSuccess
                 ? PF16_OK
                 : PF16_ERR_CUDA;
    }
    return launch_bn_fwd(b, t->x, t->gamma, t->beta, b.residual ? t->residual : nullptr, t->y,
                         t->relu_mask, t->mean, t->invstd, static_cast<uint16_t*>(ws), st) ==
                   cudaSuccess
               ? PF16_OK
               : PF16_ERR_CUDA;
  }
  const void* req[] = {t->x, t->gamma, t->mean, t->invstd, t->dy, t->dx, t->dgamma, t->dbeta};
  for (const void* p : req) {
    if (!p) return PF16_ERR_NULL;
    if (!aligned16(p)) return PF16_ERR_ALIGN;
  }
  const bool bits = b.relu && t->relu_mask;
  if (b.relu && !bits && !t->y_saved) return PF16_ERR_NULL;
  if (b.relu && !bits && !aligned16(t->y_saved)) return PF16_ERR_ALIGN;
  if (t->dresidual && !aligned16(t->dresidual)) return PF16_ERR_ALIGN;
  if (t->conv_stats && !aligned16(t->conv_stats)) return PF16_ERR_ALIGN;
  if (b.swap) {  // the swap backward reads the residual input, and takes no partial statistics
    if (!t->residual) return PF16_ERR_NULL;
    if (!aligned16(t->residual)) return PF16_ERR_ALIGN;
    if (t->conv_stats) return PF16_ERR_UNSUPPORTED;
  }
  if (device_consts(&b.status, &sms) != PF16_OK) return PF16_ERR_CUDA;
  return launch_bn_bwd(b, t->x, t->gamma, t->mean, t->invstd, t->dy,
                       b.relu && !bits ? t->y_saved : nullptr, bits ? t->relu_mask : nullptr, t->dx,
                       t->dgamma, t->dbeta, t->dresidual, static_cast<uint16_t*>(ws), st,
                       static_cast<const uint8_t*>(t->conv_stats), b.swap ? t->residual : nullptr) ==
                 cudaSuccess
             ? PF16_OK
             : PF16_ERR_CUDA;
}

int pf16_bn_relu_maxpool_fwd(const pf16_bn_desc* d, const pf16_bn_tensors* t, uint16_t* pooled,
                             uint8_t* argmax, void* ws, size_t ws_bytes, void* stream) {
  BnLaunch b;
  int rc = bn_validate(d, &b);
  if (rc != PF16_OK) return rc;
  if (!t || !pooled || !argmax) return PF16_ERR_NULL;
  if (d->flags != PF16_BN_RELU) return PF16_ERR_UNSUPPORTED;  // ReLU, no residual
  if (t->y) return PF16_ERR_ARG;                              // y is not stored
  if (bn_pool_smem_bytes(d->w, d->c) > 200 * 1024) return PF16_ERR_UNSUPPORTED;
  if (!ws) return PF16_ERR_WORKSPACE;
  if (ws_bytes < bn_ws_bytes(b)) return PF16_ERR_WORKSPACE;
  if (!aligned16(ws)) return PF16_ERR_ALIGN;
  const void* req[] = {t->x, t->gamma, t->beta, t->mean, t->invstd, pooled};
  for (const void* p : req) {
    if (!p) return PF16_ERR_NULL;
    if (!aligned16(p)) return PF16_ERR_ALIGN;
  }
  if (reinterpret_cast<uintptr_t>(argmax) % 8 != 0) return PF16_ERR_ALIGN;
  if (t->conv_stats && !aligned16(t->conv_stats)) return PF16_ERR_ALIGN;
  int sms = 0;
  if (device_consts(&b.status, &sms) != PF16_OK) return PF16_ERR_CUDA;
  return launch_bn_relu_pool_fwd(b, static_cast<const uint8_t*>(t->conv_stats), t->x, t->gamma, t->beta, t->mean,
                                 t->invstd, pooled, argmax, t->relu_mask, static_cast<uint16_t*>(ws), d->n, d->h,
                                 d->w, static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? PF16_OK
             : PF16_ERR_CUDA;
}

static int pool_check(const void* a, const void* b, int32_t n, int32_t h, int32_t w, int32_t c) {
  if (!a || !b) return PF16_ERR_NULL;
  if (!aligned16(a) || !aligned16(b)) return PF16_ERR_ALIGN;
  if (n <= 0 || h <= 0 || w <= 0 || c <= 0) return PF16_ERR_SHAPE;
  if (c % 8 != 0) return PF16_ERR_UNSUPPORTED;
  if ((long long)n * h * w * c > (1ll << 34)) return PF16_ERR_SHAPE;
  if ((long long)w * c > (1ll << 30)) return PF16_ERR_UNSUPPORTED;  // one row's index fits 32 bits
  return PF16_OK;
}

int pf16_maxpool_fwd(const uint16_t* x, uint16_t* y, int32_t n, int32_t h, int32_t w, int32_t c,
                     void* stream) {
  int rc = pool_check(x, y, n, h, w, c);
  if (rc != PF16_OK) return rc;
  return launch_maxpool_fwd(x, y, nullptr, n, h, w, c, static_cast<cudaStream_t>(stream)) ==
                 cudaSuccess
             ? PF16_OK
             : PF16_ERR_CUDA;
}

int pf16_maxpool_fwd_argmax(const uint16_t* x, uint16_t* y, uint8_t* argmax, int32_t n, int32_t h,
                            int32_t w, int32_t c, void* stream) {
  int rc = pool_check(x, y, n, h, w, c);
  if (rc != PF16_OK) return rc;
  if (!argmax) return PF16_ERR_NULL;
  if ((reinterpret_cast<uintptr_t>(argmax) & 7u) != 0) return PF16_ERR_ALIGN;
  return launch_maxpool_fwd(x, y, argmax, n, h, w, c, static_cast<cudaStream_t>(stream)) ==
                 cudaSuccess
             ? PF16_OK
             : PF16_ERR_CUDA;
}

int pf16_maxpool_bwd_argmax(const uint8_t* argmax, const uint16_t* dy, uint16_t* dx, int32_t n,
                            int32_t h, int32_t w, int32_t c, void* stream) {
  int rc = pool_check(dy, dx, n, h, w, c);
  if (rc != PF16_OK) return rc;
  if (!argmax) return PF16_ERR_NULL;
  if ((reinterpret_cast<uintptr_t>(argmax) & 7u) != 0) return PF16_ERR_ALIGN;
  return launch_maxpool_bwd_codes(argmax, dy, dx, n, h, w, c, static_cast<cudaStream_t>(stream)) ==
                 cudaSuccess
             ? PF16_OK
             : PF16_ERR_CUDA;
}

int pf16_maxpool_bwd(const uint16_t* x, const uint16_t* dy, uint16_t* dx, int32_t n, int32_t h,
                     int32_t w, int32_t c, void* stream) {
  int rc = pool_check(x, dx, n, h, w, c);
  if (rc != PF16_OK) return rc;
  if (w > 1024) return PF16_ERR_UNSUPPORTED;  // a band of 11 input rows is staged in shared memory
  if (!dy) return PF16_ERR_NULL;
  if (!aligned16(dy)) return PF16_ERR_ALIGN;
  return launch_maxpool_bwd(x, dy, dx, n, h, w, c, static_cast<cudaStream_t>(stream)) ==
                 cudaSuccess
             ? PF16_OK
             : PF16_ERR_CUDA;
}

int pf16_avgpool_fwd(const uint16_t* x, uint16_t* y, int32_t n, int32_t hw, int32_t c,
                     void* stream) {
  int rc = pool_check(x, y, n, hw, 1, c);
  if (rc != PF16_OK) return rc;
  if (hw > 4096) return PF16_ERR_UNSUPPORTED;
  return launch_avgpool_fwd(x, y, n, hw, c, static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? PF16_OK
             : PF16_ERR_CUDA;
}

int pf16_avgpool_bwd(const uint16_t* dy, uint16_t* dx, int32_t n, int32_t hw, int32_t c,
                     void* stream) {
  int rc = pool_check(dy, dx, n, hw, 1, c);
  if (rc != PF16_OK) return rc;
  return launch_avgpool_bwd(dy, dx, n, hw, c, static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? PF16_OK
             : PF16_ERR_CUDA;
}

size_t pf16_softmax_xent_workspace_size(int32_t b, int32_t k) {
  if (b <= 0 || k <= 0) return 0;
  return round_up((size_t)b * 2, 256);
}

int pf16_softmax_xent(const uint16_t* logits, const uint16_t* bias, const int32_t* labels,
                      int32_t b, int32_t k, uint16_t* loss, uint16_t* dlogits, uint16_t* dbias,
                      void* ws, size_t ws_bytes, void* stream) {
  if (!logits || !labels || !loss || !dlogits) return PF16_ERR_NULL;
  if (b <= 0 || k <= 0 || b > 65535) return PF16_ERR_SHAPE;
  if (k > 4096) return PF16_ERR_UNSUPPORTED;
  if (!ws || ws_bytes < pf16_softmax_xent_workspace_size(b, k)) return PF16_ERR_WORKSPACE;
  return launch_softmax_xent(logits, bias, labels, b, k, loss, dlogits, dbias,
                             static_cast<uint16_t*>(ws), static_cast<cudaStream_t>(stream)) ==
                 cudaSuccess
             ? PF16_OK
             : PF16_ERR_CUDA;
}

int pf16_sync_status(void* stream) {
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(st) != cudaSuccess) return PF16_ERR_CUDA;
  int* status;
  int sms;
  int rc = device_consts(&status, &sms);
  if (rc != PF16_OK) return rc;
  int v = 0;
  if (cudaMemcpy(&v, status, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
    return PF16_ERR_CUDA;
  if (v != 0) {
    const int zero = 0;
    if (cudaMemcpy(status, &zero, sizeof(int), cudaMemcpyHostToDevice) != cudaSuccess)
      return PF16_ERR_CUDA;
  }
  return v;
}

int pf16_wait_flag(const uint32_t* flag, uint32_t value, uint64_t timeout_ns, void* stream) {
  if (!flag) return PF16_ERR_NULL;
  if ((reinterpret_cast<uintptr_t>(flag) & 3u) != 0) return PF16_ERR_ALIGN;
  if (timeout_ns > 10000000000ull) return PF16_ERR_ARG;
  int* status;
  int sms;
  int rc = device_consts(&status, &sms);
  if (rc != PF16_OK) return rc;
  return launch_wait_flag(flag, value, timeout_ns, status, static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? PF16_OK
             : PF16_ERR_CUDA;
}

int pf16_tc_rate(int32_t n, int32_t f32_accum, int32_t chains, int32_t reps, double* tflops, void* stream) {
  if (!tflops) return PF16_ERR_NULL;
  if ((n != 64 && n != 128 && n != 192 && n != 256) || (f32_accum != 0 && f32_accum != 1) ||
      (chains != 1 && chains != 2) || reps < 1 || reps > (1 << 20))
    return PF16_ERR_ARG;
  int* status;
  int sms;
  int rc = device_consts(&status, &sms);
  if (rc != PF16_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const uint32_t idesc = idesc_f16(kBM, n, false, false, f32_accum != 0);
  cudaEvent_t e0, e1;
  if (cudaEventCreate(&e0) != cudaSuccess) return PF16_ERR_CUDA;
  if (cudaEventCreate(&e1) != cudaSuccess) {
    cudaEventDestroy(e0);
    return PF16_ERR_CUDA;
  }
  const unsigned long long wait_ns = 4000000000ull;
  float ms = 0.f;
  bool ok = launch_tc_rate(idesc, n, chains, reps / 4 + 1, sms, status, wait_ns, st) == cudaSuccess &&  // warm-up
            cudaEventRecord(e0, st) == cudaSuccess &&
            launch_tc_rate(idesc, n, chains, reps, sms, status, wait_ns, st) == cudaSuccess &&
            cudaEventRecord(e1, st) == cudaSuccess && cudaEventSynchronize(e1) == cudaSuccess &&
            cudaEventElapsedTime(&ms, e0, e1) == cudaSuccess;
  cudaEventDestroy(e0);
  cudaEventDestroy(e1);
  if (!ok || ms <= 0.f) return PF16_ERR_CUDA;
  const double flop = (double)sms * reps * 4.0 * 2.0 * kBM * n * 16.0;
  *tflops = flop / ((double)ms * 1e-3) / 1e12;
  return PF16_OK;
}

const char* pf16_status_string(int status) {
  switch (status) {
    case PF16_OK: return "ok";
    case PF16_ERR_NULL: return "a required pointer is NULL";
    case PF16_ERR_ALIGN: return "a tensor pointer is not 16-byte aligned";
    case PF16_ERR_SHAPE: return "invalid or inconsistent sizes";
    case PF16_ERR_UNSUPPORTED: return "sizes or options outside what the kernels support";
    case PF16_ERR_WORKSPACE: return "workspace missing or too small";
    case PF16_ERR_CUDA: return "a CUDA runtime or driver call failed";
    case PF16_ERR_TIMEOUT: return "a bounded device-side wait expired";
    case PF16_ERR_ARG: return "invalid flag, phase or enum value";
    default: return "unknown status";
  }
}

int pf16_device_arch(void) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return PF16_ERR_CUDA;
  int maj = 0, min = 0;
  if (cudaDeviceGetAttribute(&maj, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&min, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
    return PF16_ERR_CUDA;
  return maj * 10 + min;
}

uint64_t pf16_kernel_launches(void) {
  return (uint64_t)pf16::g_kernel_launches.load(std::memory_order_relaxed);
}

}  // extern "C"
