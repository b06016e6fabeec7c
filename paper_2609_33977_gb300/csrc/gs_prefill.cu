// Prefill-regime group-sparse linear (many tokens, tensor-core bound):
//   y[t, r] = sum over kept groups (r, c) of X_c[t, :] . W[r, 256c : 256c+256]   (Eq. 1)
//
// Tile = 128 tokens x 160 output rows (a "window").  For every chunk c the kept
// rows of the window form one contiguous slice of the packed tiles (rows are
// ascending inside a chunk), so the slice is a dense K-major operand that TMA
// loads as-is.  Per chunk one tcgen05 MMA chain computes D[128 tok x n] =
// X_c . W_slice^T (n <= 160 kept rows) into a TMEM scratch buffer; the
// epilogue warps then gather each window row's scratch column (or a zero
// column when the row is pruned in that chunk) into the TMEM-resident
// 128 x 160 accumulator.  W (.) M is never
// materialised and pruned groups cost neither bytes nor FLOPs.  Two scratch
// buffers let the MMA of the next slice overlap the scatter-add of this one.
//
// Roles (one CTA per SM, persistent over tiles):
//   warp 0      TMA producer (X box 128x64, W boxes of 128/64/32/16 rows)
//   warp 1      TMEM allocator + single-thread MMA issuer
//   warps 2..9  epilogue: gather-add into the accumulator, then accumulator -> bf16 y
// Each warp stages the window's per-chunk slice bounds in shared memory at the
// start of a tile; the epilogue prefetches its blocks' masks one item ahead.  Every
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
constexpr int kFW = 160;                      // output rows per tile (accumulator columns)
constexpr int kHalf = kFW / 2;                // accumulator columns owned by one epilogue warp
constexpr int kBlkRows = kWin16;              // accumulator block handled per gather round
constexpr int kBlocksPerHalf = kHalf / kBlkRows;   // 5
constexpr int kNMax = kFW;                    // kept rows per MMA item: a whole window's slice always fits
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
constexpr int kMetaInts = 2 * kMaxG;          // per warp: slice start and end per chunk
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kAccCol = 0;
constexpr uint32_t kScrCol = kFW;             // two scratch buffers of kNMax columns
constexpr uint32_t kZeroCol = kScrCol + 2 * kNMax;   // 32 columns kept at 0.0 (gather target of pruned rows)
constexpr uint64_t kWaitLimitNs = 2000000000ull;
constexpr uint64_t kDrainLimitNs = 200000000ull;
constexpr int kSmemBytes = kStages * kStageBytes + kWarps * kMetaInts * 4 + 1024;

static_assert(kZeroCol + 32 <= kTmemCols, "TMEM budget");
static_assert(kStageBytes % 1024 == 0, "stages must keep 1024-byte alignment");
static_assert(kFW % 32 == 0 && kHalf % kBlkRows == 0 && kNMax % 16 == 0, "tile shape");
static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");

struct PrefillParams {
  CUtensorMap xmap;        // x [T][in] bf16, box 64 x 128
  CUtensorMap wmap[4];     // tiles [kept][256] bf16, box 64 x {128, 64, 32, 16}
  const int32_t* win_off16;
  const uint16_t* kmask16;
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
// are packed rows [p0[c], p1[c]).
struct TileMeta {
  int32_t* p0;
  int32_t* p1;
};

__device__ __forceinline__ void load_tile_meta(const PrefillParams& P, int w, int lane, const TileMeta& M) {
  const int wlo = (kFW / kWin16) * w;
  const int whi = min(wlo + kFW / kWin16, P.nw16);
  for (int c = lane; c < P.G; c += 32) {
    const int32_t* wo = P.win_off16 + (int64_t)c * (P.nw16 + 1);
    M.p0[c] = wo[wlo];
    M.p1[c] = wo[whi];
  }
  __syncwarp();
}

// Items of a tile: the chunks whose window slice is non-empty, in order.
__device__ __forceinline__ int item_next(const PrefillParams& P, const TileMeta& M, int c) {
  for (++c; c < P.G; ++c)
    if (M.p1[c] > M.p0[c]) return c;
  return P.G;
}

// lanes 0..4 fetch (window offset, kept mask) of the five 16-row blocks of an
// epilogue warp's accumulator half for chunk c
__device__ __forceinline__ void load_blocks(const PrefillParams& P, int c, int wblk0, int lane, int& woff,
                                            uint32_t& km) {
  const int wi = wblk0 + lane;
  woff = 0;
  km = 0u;
  if (c < P.G && lane < kBlocksPerHalf && wi < P.nw16) {
    woff = __ldg(P.win_off16 + (int64_t)c * (P.nw16 + 1) + wi);
    km = __ldg(P.kmask16 + (int64_t)c * P.nw16 + wi);
  }
}

__device__ __forceinline__ void tmem_ld_x16b(uint32_t taddr, uint32_t* v) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
        "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
      : "r"(taddr)
      : "memory");
}
__device__ __forceinline__ void tmem_st_x16(uint32_t taddr, const uint32_t* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};"
      ::"r"(taddr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
        "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
      : "memory");
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
  const TileMeta M{meta_base, meta_base + kMaxG};

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
        for (int c = item_next(P, M, -1); c < P.G && ok; c = item_next(P, M, c)) {
          const int start = M.p0[c];
          const int nr = (M.p1[c] - start + 15) & ~15;
          for (int ks = 0; ks < kKSteps; ++ks) {
            if (!mbar_wait_bounded(&empty_bar[stage], phase ^ 1u, abort_flag, P.err, kWaitLimitNs,
                                   kDevErrTimeout)) {
              ok = false;
              break;
            }
            uint8_t* sx = smem + stage * kStageBytes;
            uint8_t* sw = sx + kXStageBytes;
            mbar_arrive_expect_tx(&full_bar[stage], (uint32_t)(kXStageBytes + nr * kBK * 2));
            tma_load_2d(sx, &P.xmap, &full_bar[stage], c * kGroupIn + ks * kBK, m * kBM);
            int rr = 0;
#pragma unroll
            for (int h = 0; h < 4; ++h) {
              const int hh = 128 >> h;
              while (nr - rr >= hh) {
                tma_load_2d(sw + rr * (kBK * 2), &P.wmap[h], &full_bar[stage], ks * kBK, start + rr);
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
        for (int c = item_next(P, M, -1); c < P.G && ok; c = item_next(P, M, c)) {
          const int nr = (M.p1[c] - M.p0[c] + 15) & ~15;
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
    // half h (window rows 80h .. 80h+79, five 16-row blocks).  For each item
    // (chunk) and block the warp gathers its rows' scratch columns: row i of
    // a block with kept mask m reads scratch column b0 + popc(m & (2^i - 1))
    // when kept and a column held at zero otherwise, then adds the 16 values
    // into the block with one 16-column load and store.  Every accumulator
    // column belongs to one warp, and no single-column TMEM store is needed.
    const int ew = warp - 2;
    const int q = warp & 3;
    const int h = ew >> 2;
    const uint32_t lane_off = (uint32_t)(32 * q) << 16;
    const uint32_t t_acc = tmem + lane_off + kAccCol + (uint32_t)(kHalf * h);
    const uint32_t t_scr = tmem + lane_off + kScrCol;
    const uint32_t t_zero = tmem + lane_off + kZeroCol;
    tmem_st_x32_zero(t_zero);
    int buf = 0;
    uint32_t sf_ph[2] = {0u, 0u};
    bool ok = true;
    for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x) {
      const int m = t % P.n_m, w = t / P.n_m;
      const int r0 = w * kFW + kHalf * h;
      const int wblk0 = (kFW / kWin16) * w + kBlocksPerHalf * h;
      load_tile_meta(P, w, lane, M);
      {
        const uint32_t z[16] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
#pragma unroll
        for (int k = 0; k < kBlocksPerHalf; ++k) tmem_st_x16(t_acc + kBlkRows * k, z);
      }
      tmem_wait_st();
      int c = item_next(P, M, -1);
      int woff, nwoff;
      uint32_t km, nkm;
      load_blocks(P, c, wblk0, lane, woff, km);
      while (c < P.G && ok) {
        const int cn = item_next(P, M, c);
        load_blocks(P, cn, wblk0, lane, nwoff, nkm);      // prefetch the next item's block metadata
        const int p0 = M.p0[c];
        if (!mbar_wait_bounded(&sfull_bar[buf], sf_ph[buf], abort_flag, P.err, kWaitLimitNs, kDevErrTimeout)) {
          ok = false;
          break;
        }
        sf_ph[buf] ^= 1u;
        tc_fence_after();
        const uint32_t scr = t_scr + (uint32_t)(buf * kNMax);
#pragma unroll
        for (int k = 0; k < kBlocksPerHalf; ++k) {
          const uint32_t mk = __shfl_sync(0xffffffffu, km, k);
          if (mk == 0u) continue;
          const int b0 = __shfl_sync(0xffffffffu, woff, k) - p0;   // scratch column of the block's first kept row
          const int li = lane & (kBlkRows - 1);
          const uint32_t my_addr = ((mk >> li) & 1u) ? scr + (uint32_t)(b0 + __popc(mk & ((1u << li) - 1u))) : t_zero;
          uint32_t a[kBlkRows], g[kBlkRows];
          tmem_ld_x16b(t_acc + kBlkRows * k, a);
#pragma unroll
          for (int i = 0; i < kBlkRows; ++i) g[i] = tmem_ld_x1(__shfl_sync(0xffffffffu, my_addr, i));
          tmem_wait_ld();
          reg_fence(a);
          reg_fence(g);
#pragma unroll
          for (int i = 0; i < kBlkRows; ++i) a[i] = __float_as_uint(__uint_as_float(a[i]) + __uint_as_float(g[i]));
          tmem_st_x16(t_acc + kBlkRows * k, a);
        }
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sempty_bar[buf]);
        buf ^= 1;
        c = cn;
        woff = nwoff;
        km = nkm;
      }
      if (!ok) break;
      // own accumulator half -> bf16 y rows [r0, r0 + kHalf) of token tok
      const int tok = m * kBM + 32 * q + lane;
      uint16_t* yrow = P.y + (int64_t)tok * P.out;
      const bool vec_ok = (P.out & 7) == 0;
#pragma unroll 1
      for (int col = 0; col < kHalf; col += kBlkRows) {
        uint32_t v[kBlkRows];
        tmem_ld_x16b(t_acc + col, v);
        tmem_wait_ld();
        reg_fence(v);
        const int rb = r0 + col;
        if (tok < P.T && rb < P.out) {
          if (vec_ok && rb + kBlkRows <= P.out) {
            uint4* dst = reinterpret_cast<uint4*>(yrow + rb);
#pragma unroll
            for (int u = 0; u < 2; ++u)
              dst[u] = make_uint4(pack_bf16x2(v[8 * u + 0], v[8 * u + 1]), pack_bf16x2(v[8 * u + 2], v[8 * u + 3]),
                                  pack_bf16x2(v[8 * u + 4], v[8 * u + 5]), pack_bf16x2(v[8 * u + 6], v[8 * u + 7]));
          } else {
#pragma unroll
            for (int i = 0; i < kBlkRows; ++i)
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
  P.win_off16 = p->win_off16;
  P.kmask16 = p->kmask16;
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
