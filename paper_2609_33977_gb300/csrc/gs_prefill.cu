// Prefill-regime group-sparse linear (many tokens, tensor-core bound):
//   y[t, r] = sum over kept groups (r, c) of X_c[t, :] . W[r, 256c : 256c+256]   (Eq. 1)
//
// Tile = 128 tokens x 192 output rows (a "window").  For every chunk c the kept
// rows of the window form one contiguous slice of the packed tiles (rows are
// ascending inside a chunk), so the slice is a dense K-major operand that TMA
// loads as-is.  Per (chunk, slice of <= 160 kept rows) one tcgen05 MMA chain
// computes D[128 tok x n] = X_c . W_slice^T into a TMEM scratch buffer; the
// epilogue warps then add scratch column j into accumulator column
// row_idx[j] - 192*window (TMEM-resident, 192 columns).  W (.) M is never
// materialised and pruned groups cost neither bytes nor FLOPs.  Two scratch
// buffers let the MMA of the next slice overlap the scatter-add of this one.
//
// Roles (one CTA per SM, persistent over tiles):
//   warp 0      TMA producer (X box 128x64, W boxes of 128/64/32/16 rows)
//   warp 1      TMEM allocator + single-thread MMA issuer
//   warps 2..9  epilogue: scatter-add, then accumulator -> bf16 y
// Each warp stages the window's per-chunk slice bounds in shared memory at the
// start of a tile, so no role waits on global metadata per item.  Every
// mbarrier wait is bounded; a wait that runs out raises a CTA-wide abort flag
// and the library's device error flag, and all roles wind down.
#include "gs_common.cuh"
#include "gs_sm100.cuh"

#include <cuda.h>
#include <cstring>
#include <mutex>

namespace gs {
namespace {
using namespace sm100;

constexpr int kBM = 128;                      // tokens per tile (TMEM lanes)
constexpr int kFW = 192;                      // output rows per tile (accumulator columns)
constexpr int kHalf = kFW / 2;                // accumulator columns owned by one epilogue warp
constexpr int kNMax = 160;                    // kept rows per MMA item (scratch columns)
constexpr int kBK = 64;                       // k per pipeline stage: one 128-byte swizzle row
constexpr int kKSteps = kGroupIn / kBK;       // 4 stages per 256-wide chunk
constexpr int kStages = 5;
constexpr int kXStageBytes = kBM * kBK * 2;   // 16 KB
constexpr int kWStageBytes = kNMax * kBK * 2; // 20 KB
constexpr int kStageBytes = kXStageBytes + kWStageBytes;
constexpr int kEpiWarps = 8;
constexpr int kWarps = 2 + kEpiWarps;
constexpr int kThreads = kWarps * 32;
constexpr int kMaxG = 256;                    // chunks per layer handled by this kernel (in <= 65536)
constexpr int kMetaInts = 3 * kMaxG;          // per warp: slice start, end, and first row of the upper half
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kAccCol = 0;
constexpr uint32_t kScrCol = kFW;             // two scratch buffers of kNMax columns
constexpr uint64_t kWaitLimitNs = 2000000000ull;
constexpr uint64_t kDrainLimitNs = 200000000ull;
constexpr int kSmemBytes = kStages * kStageBytes + kWarps * kMetaInts * 4 + 1024;

static_assert(kScrCol + 2 * kNMax <= kTmemCols, "TMEM budget");
static_assert(kStageBytes % 1024 == 0, "stages must keep 1024-byte alignment");
static_assert(kFW % 16 == 0 && kHalf % 32 == 0 && kNMax % 32 == 0, "tile shape");
static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");

struct PrefillParams {
  CUtensorMap xmap;        // x [T][in] bf16, box 64 x 128
  CUtensorMap wmap[4];     // tiles [kept][256] bf16, box 64 x {128, 64, 32, 16}
  const int32_t* row_idx;
  const int32_t* win_off16;
  uint16_t* y;
  int32_t out, G, nw16, T;
  int32_t n_m, n_w;
  int* err;
};

__device__ __forceinline__ uint32_t pack_bf16x2(uint32_t lo, uint32_t hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(__uint_as_float(lo), __uint_as_float(hi));
  return *reinterpret_cast<const uint32_t*>(&h);
}

// Per-warp copy of a tile's slice bounds: for chunk c the window's kept rows
// are packed rows [p0[c], p1[c]); rows of the upper accumulator half start at pm[c].
struct TileMeta {
  int32_t* p0;
  int32_t* p1;
  int32_t* pm;
};

__device__ __forceinline__ void load_tile_meta(const PrefillParams& P, int w, int lane, const TileMeta& M) {
  const int wlo = (kFW / kWin16) * w;
  const int whi = min(wlo + kFW / kWin16, P.nw16);
  const int wmid = min(wlo + kHalf / kWin16, P.nw16);
  for (int c = lane; c < P.G; c += 32) {
    const int32_t* wo = P.win_off16 + (int64_t)c * (P.nw16 + 1);
    M.p0[c] = wo[wlo];
    M.p1[c] = wo[whi];
    M.pm[c] = wo[wmid];
  }
  __syncwarp();
}

// Items of a tile: chunk c = 0..G-1, slice cut into pieces of <= kNMax rows.
struct Item {
  int c, start, end;
};
__device__ __forceinline__ bool item_scan(const PrefillParams& P, const TileMeta& M, int c0, Item& it) {
  for (int c = c0; c < P.G; ++c) {
    const int p0 = M.p0[c], p1 = M.p1[c];
    if (p1 > p0) {
      it.c = c;
      it.start = p0;
      it.end = p1;
      return true;
    }
  }
  return false;
}
__device__ __forceinline__ bool item_next(const PrefillParams& P, const TileMeta& M, Item& it) {
  if (it.start + kNMax < it.end) {
    it.start += kNMax;
    return true;
  }
  return item_scan(P, M, it.c + 1, it);
}

// lane l receives the output rows of item columns l, 32+l, ..., 128+l
__device__ __forceinline__ void load_dst(const PrefillParams& P, const Item& it, bool have, int lane,
                                         int (&d)[kNMax / 32]) {
#pragma unroll
  for (int b = 0; b < kNMax / 32; ++b) {
    const int j = it.start + 32 * b + lane;
    d[b] = (have && j < it.end && j < it.start + kNMax) ? __ldg(P.row_idx + j) : 0;
  }
}

__global__ void __launch_bounds__(kThreads, 1) k_prefill(const __grid_constant__ PrefillParams P) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kStages];
  __shared__ __align__(8) uint64_t empty_bar[kStages];
  __shared__ __align__(8) uint64_t sfull_bar[2];
  __shared__ __align__(8) uint64_t sempty_bar[2];
  __shared__ __align__(8) uint64_t drain_bar;
  __shared__ uint32_t tmem_base_s;
  __shared__ int abort_s;

  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int32_t* meta_base = reinterpret_cast<int32_t*>(smem + kStages * kStageBytes) + warp * kMetaInts;
  const TileMeta M{meta_base, meta_base + kMaxG, meta_base + 2 * kMaxG};

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&sfull_bar[b], 1);
      mbar_init(&sempty_bar[b], kEpiWarps);
    }
    mbar_init(&drain_bar, 1);
    abort_s = 0;
    fence_mbar_init();
    prefetch_tmap(&P.xmap);
    for (int h = 0; h < 4; ++h) prefetch_tmap(&P.wmap[h]);
  }
  if (warp == 1) {
    tmem_alloc(&tmem_base_s, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  volatile int* abort_flag = &abort_s;
  const int n_tiles = P.n_m * P.n_w;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    uint32_t stage = 0, phase = 0;
    int armed[kStages];
    for (int s = 0; s < kStages; ++s) armed[s] = -1;
    bool ok = true;
    for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x) {
      const int m = t % P.n_m, w = t / P.n_m;
      load_tile_meta(P, w, lane, M);
      if (lane == 0) {
        Item it;
        bool have = item_scan(P, M, 0, it);
        for (; have && ok; have = item_next(P, M, it)) {
          const int n = min(kNMax, it.end - it.start);
          const int nr = (n + 15) & ~15;
          for (int ks = 0; ks < kKSteps; ++ks) {
            if (!mbar_wait_bounded(&empty_bar[stage], phase ^ 1u, abort_flag, P.err, kWaitLimitNs,
                                   kDevErrTimeout)) {
              ok = false;
              break;
            }
            uint8_t* sx = smem + stage * kStageBytes;
            uint8_t* sw = sx + kXStageBytes;
            mbar_arrive_expect_tx(&full_bar[stage], (uint32_t)(kXStageBytes + nr * kBK * 2));
            tma_load_2d(sx, &P.xmap, &full_bar[stage], it.c * kGroupIn + ks * kBK, m * kBM);
            int rr = 0;
#pragma unroll
            for (int h = 0; h < 4; ++h) {
              const int hh = 128 >> h;
              while (nr - rr >= hh) {
                tma_load_2d(sw + rr * (kBK * 2), &P.wmap[h], &full_bar[stage], ks * kBK, it.start + rr);
                rr += hh;
              }
            }
            armed[stage] = (int)phase;
            if (++stage == kStages) {
              stage = 0;
              phase ^= 1u;
            }
          }
        }
      }
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
    }
    if (lane == 0 && !ok) {
      // let copies already in flight land before the CTA retires
      for (int s = 0; s < kStages; ++s) {
        if (armed[s] < 0) continue;
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait(&full_bar[s], (uint32_t)armed[s]))
          if (globaltimer_ns() - t0 > kDrainLimitNs) break;
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    uint32_t stage = 0, phase = 0;
    int buf = 0;
    uint32_t se_ph[2] = {0u, 0u};
    bool ok = true;
    for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x) {
      const int w = t / P.n_m;
      load_tile_meta(P, w, lane, M);
      if (lane == 0) {
        Item it;
        bool have = item_scan(P, M, 0, it);
        for (; have && ok; have = item_next(P, M, it)) {
          const int n = min(kNMax, it.end - it.start);
          const int nr = (n + 15) & ~15;
          if (!mbar_wait_bounded(&sempty_bar[buf], se_ph[buf] ^ 1u, abort_flag, P.err, kWaitLimitNs,
                                 kDevErrTimeout)) {
            ok = false;
            break;
          }
          se_ph[buf] ^= 1u;
          tc_fence_after();
          const uint32_t d = tmem + kScrCol + (uint32_t)(buf * kNMax);
          const uint32_t idesc = idesc_bf16_f32(kBM, nr);
          for (int ks = 0; ks < kKSteps; ++ks) {
            if (!mbar_wait_bounded(&full_bar[stage], phase, abort_flag, P.err, kWaitLimitNs, kDevErrTimeout)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t sx = smem_u32(smem + stage * kStageBytes);
            const uint64_t ad = sdesc_sw128(sx);
            const uint64_t bd = sdesc_sw128(sx + kXStageBytes);
#pragma unroll
            for (int kk = 0; kk < kBK / 16; ++kk)
              mma_bf16_ss(d, ad + (uint64_t)(2 * kk), bd + (uint64_t)(2 * kk), idesc, (ks | kk) != 0 ? 1u : 0u);
            mma_commit(&empty_bar[stage]);
            if (++stage == kStages) {
              stage = 0;
              phase ^= 1u;
            }
          }
          if (!ok) break;
          mma_commit(&sfull_bar[buf]);
          buf ^= 1;
        }
      }
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
    }
    if (lane == 0) {
      // all MMAs issued by this thread have completed once drain_bar flips
      mma_commit(&drain_bar);
      mbar_wait_bounded(&drain_bar, 0u, nullptr, P.err, kWaitLimitNs, kDevErrTimeout);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue
    // Warp (q, h): TMEM lane quarter q (tokens 32q..32q+31) and accumulator
    // half h (columns kHalf*h .. kHalf*h + kHalf - 1, window rows likewise).
    // Kept rows are ascending inside an item, so the item's columns landing in
    // half 0 are a prefix [0, jsplit) and the rest land in half 1: every
    // accumulator column is only ever touched by one warp.
    const int ew = warp - 2;
    const int q = warp & 3;
    const int h = ew >> 2;
    const uint32_t lane_off = (uint32_t)(32 * q) << 16;
    const uint32_t t_acc = tmem + lane_off + kAccCol;
    const uint32_t t_scr = tmem + lane_off + kScrCol;
    int buf = 0;
    uint32_t sf_ph[2] = {0u, 0u};
    bool ok = true;
    for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x) {
      const int m = t % P.n_m, w = t / P.n_m;
      const int r0 = w * kFW;
      load_tile_meta(P, w, lane, M);
#pragma unroll
      for (int col = 0; col < kHalf; col += 32) tmem_st_x32_zero(t_acc + kHalf * h + col);
      tmem_wait_st();
      Item it;
      bool have = item_scan(P, M, 0, it);
      int dreg[kNMax / 32];
      load_dst(P, it, have, lane, dreg);
      while (have && ok) {
        Item nx = it;
        const bool have_nx = item_next(P, M, nx);
        int ndreg[kNMax / 32];
        load_dst(P, nx, have_nx, lane, ndreg);            // prefetch the next item's rows
        const int n = min(kNMax, it.end - it.start);
        const int jsplit = min(max(M.pm[it.c] - it.start, 0), n);
        const int jlo = h ? jsplit : 0, jhi = h ? n : jsplit;
        if (!mbar_wait_bounded(&sfull_bar[buf], sf_ph[buf], abort_flag, P.err, kWaitLimitNs, kDevErrTimeout)) {
          ok = false;
          break;
        }
        sf_ph[buf] ^= 1u;
        tc_fence_after();
        const uint32_t scr = t_scr + (uint32_t)(buf * kNMax);
#pragma unroll
        for (int b = 0; b < kNMax / 32; ++b) {
          if (32 * b + 32 <= jlo || 32 * b >= jhi) continue;
          uint32_t sv[32], av[32], col[32];
          tmem_ld_x32(scr + (uint32_t)(32 * b), sv);
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            col[j] = (uint32_t)(__shfl_sync(0xffffffffu, dreg[b], j) - r0);
            av[j] = 0u;
            if (32 * b + j >= jlo && 32 * b + j < jhi) av[j] = tmem_ld_x1(t_acc + col[j]);
          }
          tmem_wait_ld();
          reg_fence(sv);
          reg_fence(av);
#pragma unroll
          for (int j = 0; j < 32; ++j)
            if (32 * b + j >= jlo && 32 * b + j < jhi)
              tmem_st_x1(t_acc + col[j], __float_as_uint(__uint_as_float(av[j]) + __uint_as_float(sv[j])));
        }
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sempty_bar[buf]);
        buf ^= 1;
        it = nx;
        have = have_nx;
#pragma unroll
        for (int b = 0; b < kNMax / 32; ++b) dreg[b] = ndreg[b];
      }
      if (!ok) break;
      // own accumulator half -> bf16 y rows [r0 + kHalf*h, r0 + kHalf*h + kHalf) of token tok
      const int tok = m * kBM + 32 * q + lane;
      uint16_t* yrow = P.y + (int64_t)tok * P.out;
      const bool vec_ok = (P.out & 7) == 0;
#pragma unroll 1
      for (int col = 0; col < kHalf; col += 32) {
        uint32_t v[32];
        tmem_ld_x32(t_acc + kHalf * h + col, v);
        tmem_wait_ld();
        reg_fence(v);
        const int rb = r0 + kHalf * h + col;
        if (tok < P.T && rb < P.out) {
          if (vec_ok && rb + 32 <= P.out) {
            uint4* dst = reinterpret_cast<uint4*>(yrow + rb);
#pragma unroll
            for (int u = 0; u < 4; ++u)
              dst[u] = make_uint4(pack_bf16x2(v[8 * u + 0], v[8 * u + 1]), pack_bf16x2(v[8 * u + 2], v[8 * u + 3]),
                                  pack_bf16x2(v[8 * u + 4], v[8 * u + 5]), pack_bf16x2(v[8 * u + 6], v[8 * u + 7]));
          } else {
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (rb + i < P.out) yrow[rb + i] = __bfloat16_as_ushort(__float2bfloat16_rn(__uint_as_float(v[i])));
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ------------------------------------------------------------------ host side
int sm_count() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 148;
  }
  return n;
}

}  // namespace

gs_status prefill_prepare_weight_maps(gs_packed* p) {
  p->wmaps_valid = false;
  if (p->kept == 0) return GS_OK;
  static_assert(sizeof(CUtensorMap) == 128, "CUtensorMap size");
  for (int h = 0; h < 4; ++h) {
    CUtensorMap m;
    if (!encode_tmap_2d_bf16(&m, p->tiles, kGroupIn, (uint64_t)p->kept, kBK, (uint32_t)(128 >> h), true))
      return GS_ERR_CUDA;
    std::memcpy(p->wmaps[h], &m, sizeof(m));
  }
  p->wmaps_valid = true;
  return GS_OK;
}

int prefill_max_chunks() { return kMaxG; }

gs_status launch_prefill(const void* x, const gs_packed* p, int64_t T, void* y, cudaStream_t s) {
  if (T <= 0) return GS_OK;
  if (p->kept == 0) {
    return cudaMemsetAsync(y, 0, (size_t)T * (size_t)p->out * 2, s) == cudaSuccess ? GS_OK : GS_ERR_CUDA;
  }
  if (!p->wmaps_valid) return GS_ERR_CUDA;
  if (p->G > kMaxG) return GS_ERR_UNSUPPORTED;
  static std::once_flag attr_once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(attr_once, []() {
    attr_err = cudaFuncSetAttribute(k_prefill, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
  });
  if (attr_err != cudaSuccess) return GS_ERR_CUDA;

  PrefillParams P;
  std::memset(&P, 0, sizeof(P));
  if (!encode_tmap_2d_bf16(&P.xmap, x, (uint64_t)p->in, (uint64_t)T, kBK, kBM, true)) return GS_ERR_CUDA;
  for (int h = 0; h < 4; ++h) std::memcpy(&P.wmap[h], p->wmaps[h], sizeof(CUtensorMap));
  P.row_idx = p->row_idx;
  P.win_off16 = p->win_off16;
  P.y = static_cast<uint16_t*>(y);
  P.out = (int32_t)p->out;
  P.G = p->G;
  P.nw16 = p->nw16;
  P.T = (int32_t)T;
  P.n_m = (int32_t)((T + kBM - 1) / kBM);
  P.n_w = (int32_t)((p->out + kFW - 1) / kFW);
  P.err = device_error_flag();
  if (!P.err) return GS_ERR_CUDA;
  const int64_t tiles = (int64_t)P.n_m * P.n_w;
  const int grid = (int)(tiles < sm_count() ? tiles : sm_count());
  k_prefill<<<grid, kThreads, kSmemBytes, s>>>(P);
  note_launch();
  return cudaGetLastError() == cudaSuccess ? GS_OK : GS_ERR_CUDA;
}

}  // namespace gs
