// Prefill-regime group-sparse linear (many tokens, tensor-core bound):
//   y[t, r] = sum over kept groups (r, c) of X_c[t, :] . W[r, 256c : 256c+256]   (Eq. 1)
//
// Tile = 128 tokens x 256 output rows (a "window").  For every chunk c the kept
// rows of the window form one contiguous slice of the packed tiles (rows are
// ascending inside a chunk), so the slice is a dense K-major operand that TMA
// can load as-is.  Per (chunk, slice of <= 128 kept rows) one tcgen05 MMA
// chain computes D[128 tok x n] = X_c . W_slice^T into a TMEM scratch buffer;
// the epilogue warps then add each scratch column j into accumulator column
// row_idx[j] - 256*window (TMEM-resident, 256 columns).  W (.) M is never
// materialised and pruned groups cost neither bytes nor FLOPs.  Two scratch
// buffers let the MMA of the next slice overlap the scatter-add of this one.
//
// Roles (one CTA per SM, persistent over tiles):
//   warp 0      TMA producer (X box 128x64, W boxes of 128/64/32/16 rows)
//   warp 1      TMEM allocator + single-thread MMA issuer
//   warps 2..5  epilogue: scatter-add, then accumulator -> bf16 y
// Every mbarrier wait is bounded; a wait that runs out raises a CTA-wide abort
// flag and the library's device error flag, and all roles wind down.
#include "gs_common.cuh"
#include "gs_sm100.cuh"

#include <cuda.h>
#include <cstring>
#include <mutex>

namespace gs {
namespace {
using namespace sm100;

constexpr int kBM = 128;                      // tokens per tile (TMEM lanes)
constexpr int kFW = 256;                      // output rows per tile (accumulator columns)
constexpr int kNMax = 128;                    // kept rows per MMA item (scratch columns)
constexpr int kBK = 64;                       // k per pipeline stage: one 128-byte swizzle row
constexpr int kKSteps = kGroupIn / kBK;       // 4 stages per 256-wide chunk
constexpr int kStages = 6;
constexpr int kXStageBytes = kBM * kBK * 2;   // 16 KB
constexpr int kWStageBytes = kNMax * kBK * 2; // 16 KB
constexpr int kStageBytes = kXStageBytes + kWStageBytes;
constexpr int kEpiWarps = 4;
constexpr int kThreads = (2 + kEpiWarps) * 32;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kAccCol = 0;
constexpr uint32_t kScrCol = kFW;             // two scratch buffers of kNMax columns
constexpr uint64_t kWaitLimitNs = 2000000000ull;
constexpr uint64_t kDrainLimitNs = 200000000ull;
constexpr int kSmemBytes = kStages * kStageBytes + 1024;

static_assert(kScrCol + 2 * kNMax <= kTmemCols, "TMEM budget");

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
    if (lane == 0) {
      uint32_t stage = 0, phase = 0;
      int armed[kStages];
      for (int s = 0; s < kStages; ++s) armed[s] = -1;
      bool ok = true;
      for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x) {
        const int m = t % P.n_m, w = t / P.n_m;
        const int wlo = 16 * w, whi = min(16 * w + 16, P.nw16);
        for (int c = 0; c < P.G && ok; ++c) {
          const int32_t* wo = P.win_off16 + (int64_t)c * (P.nw16 + 1);
          const int p0 = wo[wlo], p1 = wo[whi];
          for (int start = p0; start < p1 && ok; start += kNMax) {
            const int n = min(kNMax, p1 - start);
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
              tma_load_2d(sx, &P.xmap, &full_bar[stage], c * kGroupIn + ks * kBK, m * kBM);
              int rr = 0;
#pragma unroll
              for (int h = 0; h < 4; ++h) {
                const int hh = kNMax >> h;
                if (nr - rr >= hh) {
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
      }
      if (!ok) {
        // let copies already in flight land before the CTA retires
        for (int s = 0; s < kStages; ++s) {
          if (armed[s] < 0) continue;
          const uint64_t t0 = globaltimer_ns();
          while (!mbar_try_wait(&full_bar[s], (uint32_t)armed[s]))
            if (globaltimer_ns() - t0 > kDrainLimitNs) break;
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      uint32_t stage = 0, phase = 0;
      int buf = 0;
      uint32_t se_ph[2] = {0u, 0u};
      bool ok = true;
      for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x) {
        const int w = t / P.n_m;
        const int wlo = 16 * w, whi = min(16 * w + 16, P.nw16);
        for (int c = 0; c < P.G && ok; ++c) {
          const int32_t* wo = P.win_off16 + (int64_t)c * (P.nw16 + 1);
          const int p0 = wo[wlo], p1 = wo[whi];
          for (int start = p0; start < p1 && ok; start += kNMax) {
            const int n = min(kNMax, p1 - start);
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
      }
      // all MMAs issued by this thread have completed once drain_bar flips
      mma_commit(&drain_bar);
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(&drain_bar, 0u))
        if (globaltimer_ns() - t0 > kWaitLimitNs) {
          *abort_flag = 1;
          atomicExch(P.err, kDevErrTimeout);
          break;
        }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;
    const uint32_t lane_off = (uint32_t)(32 * q) << 16;
    const uint32_t t_acc = tmem + lane_off + kAccCol;
    const uint32_t t_scr = tmem + lane_off + kScrCol;
    int buf = 0;
    uint32_t sf_ph[2] = {0u, 0u};
    bool ok = true;
    for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x) {
      const int m = t % P.n_m, w = t / P.n_m;
      const int wlo = 16 * w, whi = min(16 * w + 16, P.nw16);
      const int r0 = w * kFW;
#pragma unroll
      for (int col = 0; col < kFW; col += 32) tmem_st_x32_zero(t_acc + col);
      tmem_wait_st();
      for (int c = 0; c < P.G && ok; ++c) {
        const int32_t* wo = P.win_off16 + (int64_t)c * (P.nw16 + 1);
        const int p0 = wo[wlo], p1 = wo[whi];
        for (int start = p0; start < p1; start += kNMax) {
          const int n = min(kNMax, p1 - start);
          if (!mbar_wait_bounded(&sfull_bar[buf], sf_ph[buf], abort_flag, P.err, kWaitLimitNs, kDevErrTimeout)) {
            ok = false;
            break;
          }
          sf_ph[buf] ^= 1u;
          tc_fence_after();
          const uint32_t scr = t_scr + (uint32_t)(buf * kNMax);
          for (int j0 = 0; j0 < n; j0 += 16) {
            const int nn = min(16, n - j0);
            uint32_t sv[16];
            tmem_ld_x16(scr + (uint32_t)j0, sv);
            uint32_t dc[16], av[16];
#pragma unroll
            for (int jj = 0; jj < 16; ++jj) {
              dc[jj] = jj < nn ? (uint32_t)(__ldg(P.row_idx + start + j0 + jj) - r0) : 0u;
              av[jj] = 0u;
            }
#pragma unroll
            for (int jj = 0; jj < 16; ++jj)
              if (jj < nn) av[jj] = tmem_ld_x1(t_acc + dc[jj]);
            tmem_wait_ld();
            reg_fence(sv);
            reg_fence(av);
#pragma unroll
            for (int jj = 0; jj < 16; ++jj)
              if (jj < nn)
                tmem_st_x1(t_acc + dc[jj], __float_as_uint(__uint_as_float(av[jj]) + __uint_as_float(sv[jj])));
          }
          tmem_wait_st();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&sempty_bar[buf]);
          buf ^= 1;
        }
      }
      if (!ok) break;
      // accumulator -> bf16 y rows [r0, r0+256) of token tok
      const int tok = m * kBM + 32 * q + lane;
      uint16_t* yrow = P.y + (int64_t)tok * P.out;
      const bool vec_ok = (P.out & 7) == 0;
#pragma unroll 1
      for (int col = 0; col < kFW; col += 32) {
        uint32_t v[32];
        tmem_ld_x32(t_acc + col, v);
        tmem_wait_ld();
        reg_fence(v);
        const int rb = r0 + col;
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
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, []() {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  });
  return fn;
}

bool encode_2d_bf16(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer, uint32_t box_inner,
                    uint32_t box_outer) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {inner, outer};
  const cuuint64_t strides[1] = {inner * 2};
  const cuuint32_t box[2] = {box_inner, box_outer};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

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
    if (!encode_2d_bf16(&m, p->tiles, kGroupIn, (uint64_t)p->kept, kBK, (uint32_t)(kNMax >> h)))
      return GS_ERR_CUDA;
    std::memcpy(p->wmaps[h], &m, sizeof(m));
  }
  p->wmaps_valid = true;
  return GS_OK;
}

gs_status launch_prefill(const void* x, const gs_packed* p, int64_t T, void* y, cudaStream_t s) {
  if (T <= 0) return GS_OK;
  if (p->kept == 0) {
    return cudaMemsetAsync(y, 0, (size_t)T * (size_t)p->out * 2, s) == cudaSuccess ? GS_OK : GS_ERR_CUDA;
  }
  if (!p->wmaps_valid) return GS_ERR_CUDA;
  static std::once_flag attr_once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(attr_once, []() {
    attr_err = cudaFuncSetAttribute(k_prefill, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
  });
  if (attr_err != cudaSuccess) return GS_ERR_CUDA;

  PrefillParams P;
  std::memset(&P, 0, sizeof(P));
  if (!encode_2d_bf16(&P.xmap, x, (uint64_t)p->in, (uint64_t)T, kBK, kBM)) return GS_ERR_CUDA;
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
