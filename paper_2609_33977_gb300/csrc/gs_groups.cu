// Square g x g groups (Sec. 2.1 with g_out = g_in = g; the Sec. 3.5 ablation
// and App. E evaluate g = 16, 32, 64 and 128): packing, unpacking and the
// group-sparse linear y = x (W (.) M)^T with M = B (x) 1_{g x g} (Eq. 1).
//
// Packed layout (the same sequential definition as the 1 x 256 layout, per
// column block): column block v (input columns [g v, g v + g)) owns packed
// tiles [offsets[v], offsets[v + 1]); inside a column block the kept block
// rows u ascend; tile j is the g x g block of W at rows g u.., columns g v..,
// row-major, a bit copy, and row_idx[j] = u.  Per (column block, window of
// 128 output rows) the library also keeps the first tile of the window's
// slice and a bitmask of its kept block rows.
//
// Linear.  A unit of work is 128 tokens x one window of 128 output rows,
// R = 128 / g block rows.  In column block v the window's kept tiles are one
// contiguous slice of the packed tiles, i.e. a dense [n g x g] matrix that
// one TMA box loads, next to one box of the 128 tokens' x columns of v.  Each
// kept tile is a whole tensor-core operand: its MMAs (M = 128 tokens, N = g
// rows, K = g) accumulate straight into its block row's g columns of a
// 128-column TMEM accumulator, so nothing is gathered or scattered, and the
// accumulator is read once per unit.  Pruned tiles cost neither bytes nor
// FLOPs.  Token rows beyond T read as zero (TMA fill) and are not stored; the
// same kernel serves every token count.
//
// For T < 128 the x boxes hold only T rows: the accumulator rows of the other
// tokens then add up whatever the stage held before, and are never stored.
//
// Above 128 tokens a cluster of two CTAs owns a 256-token unit (one SM per 128
// tokens, M = 256 MMAs issued by the leader, each CTA loading its own tokens'
// x and one half of every tile's rows), which halves both the MMA instructions
// and the W bytes each SM handles.
//
// Roles (one CTA per SM, persistent over units): warp 0 TMA producer, warp 1
// TMEM allocator + single-thread MMA issuer, warps 2..5 epilogue (warp w reads
// TMEM lanes 32 (w % 4) ..).  Two accumulator buffers let the epilogue of one
// unit overlap the MMAs of the next.  Shared-memory operands use the swizzle
// whose width is one operand row: 32 B (g = 16), 64 B (g = 32), 128 B
// (g = 64; g = 128 as two 64-column slabs).  Every mbarrier wait is bounded;
// a wait that runs out raises the CTA's abort flag and the library's device
// error flag, and every role winds down.
#include "gs_common.cuh"
#include "gs_sm100.cuh"

#include <cuda.h>
#include <algorithm>
#include <cstring>
#include <mutex>
#include <vector>

namespace gs {
namespace {
using namespace sm100;

constexpr int kSqM = 128;                 // tokens per unit (TMEM lanes)
constexpr int kSqWin = 128;               // output rows per window (accumulator columns)
constexpr int kSqAccBufs = 2;
constexpr uint32_t kSqTmemCols = kSqAccBufs * kSqWin;
constexpr int kSqEpiWarps = 4;
constexpr int kSqThreads = (2 + kSqEpiWarps) * 32;
constexpr int kSqMaxLayers = 8;
constexpr int kSqDenseMaxG = 64;          // above the decode regime, g <= this takes the zero-filled kernel (7B block, T = 2048: 64x64 525 vs 476 TFLOP/s)
constexpr int kSqDecodeMaxTokensZf = 32;  // decode regime of the layers the zero-filled kernel takes
constexpr int kSqMaxMaps = 8;             // W slice heights g, 2g, ..., R g (R <= 8)
constexpr uint64_t kSqWaitLimitNs = 2000000000ull;
constexpr uint64_t kSqDrainLimitNs = 200000000ull;

template <int G, bool kPair>
struct Sq {
  static constexpr int R = kSqWin / G;                  // block rows per window
  static constexpr int kSlabs = G > 64 ? 2 : 1;         // 64-column slabs per operand row
  static constexpr int kRowB = G >= 64 ? 128 : 2 * G;   // operand row bytes within a slab = swizzle width
  static constexpr int kSlab = 128 * kRowB;             // x slab: 128 token rows at the swizzle pitch
  static constexpr int kRegion = kSlabs * kSlab;        // x bytes per stage
  static constexpr int kWRows = kPair ? kSqWin / 2 : kSqWin;   // W rows a CTA holds per stage (pair: half of each tile)
  static constexpr int kWSlab = kWRows * kRowB;
  static constexpr int kWRegion = kSlabs * kWSlab;
  static constexpr int kStageBytes = ((kRegion + kWRegion) + 1023) / 1024 * 1024;
  // as many stages as fit: a stage is one column block's copies, and the
  // copies of one stage wait for the MMAs of the stage before its last use,
  // so small groups need many stages in flight to cover the round trip
  static constexpr int kStages = (200 * 1024) / kStageBytes > 32 ? 32 : (200 * 1024) / kStageBytes;
  static constexpr uint32_t kSwz = G >= 64 ? 2u : (G == 32 ? 4u : 6u);   // UMMA layout: 128 / 64 / 32-byte swizzle
  static constexpr uint32_t kSBO = 8 * kRowB;           // bytes between 8-row core groups
  static constexpr int kKSteps = G / 16;
  static constexpr int kTile = kPair ? 2 * kSqM : kSqM; // tokens per unit
  static constexpr int kSmem = kStages * kStageBytes + 2 * 32 * 8 + 1024;
  static_assert(R >= 1 && R <= kSqMaxMaps, "window holds 1..8 block rows");
  static_assert(kSmem <= 227 * 1024, "shared memory budget");
  static_assert(kRegion % 1024 == 0, "the W region keeps 1024-byte alignment");
};

struct SqLayer {
  CUtensorMap xmap;                  // x [T][in]: box g x min(T, 128) rows (g = 128: one 64-wide slab)
  CUtensorMap wmap[kSqMaxMaps];      // tiles as [K g][g]: box heights g, 2g, ..., R g
  const int32_t* gwoff;              // [Gin][nwin + 1]
  const uint8_t* gwmask;             // [Gin][nwin]
  uint16_t* y;
  int32_t out, Gin, nwin, n_m, tile_begin;
};
struct SqParams {
  SqLayer L[kSqMaxLayers];
  int32_t n_layers, T, n_tiles;
  int32_t x_rows;            // rows of each x box: min(T, 128) (token rows past it hold stale data, never stored)
  int* err;
  TileList tl;               // which owner takes which tiles
};

__device__ __forceinline__ int sq_layer_of(const SqParams& P, int t) {
  int l = 0;
  while (l + 1 < P.n_layers && P.L[l + 1].tile_begin <= t) ++l;
  return l;
}

// UMMA shared-memory descriptor, K-major operand with the given swizzle
// (layout type 2 / 4 / 6 = 128 / 64 / 32 bytes) and 8-row group stride.
__device__ __forceinline__ uint64_t sq_desc(uint32_t saddr, uint32_t sbo, uint32_t swz) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
  d |= (uint64_t)1 << 16;                          // leading byte offset (unused for swizzled K-major)
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;     // stride byte offset
  d |= (uint64_t)1 << 46;                          // descriptor version
  d |= (uint64_t)swz << 61;
  return d;
}

// One round of a unit's items: column blocks c0 .. c0 + 31 whose window slice is
// non-empty, written to buf in order as {v | n << 16 | mask << 24, first tile}.
__device__ __forceinline__ int sq_items(const SqLayer& L, int w, int c0, int lane, uint2* buf) {
  const int v = c0 + lane;
  int p0 = 0, p1 = 0;
  uint32_t mk = 0u;
  if (v < L.Gin) {
    const int32_t* wo = L.gwoff + (int64_t)v * (L.nwin + 1);
    p0 = wo[w];
    p1 = wo[w + 1];
    mk = L.gwmask[(int64_t)v * L.nwin + w];
  }
  const bool ne = p1 > p0;
  const uint32_t ballot = __ballot_sync(0xffffffffu, ne);
  if (ne) buf[__popc(ballot & ((1u << lane) - 1u))] = make_uint2((uint32_t)v | ((uint32_t)(p1 - p0) << 16) | (mk << 24),
                                                                 (uint32_t)p0);
  __syncwarp();
  return __popc(ballot);
}

__device__ __forceinline__ uint32_t sq_pack_bf16x2(float lo, float hi, bool keep) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(keep ? lo : 0.f, keep ? hi : 0.f);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// kPair: a cluster of two CTAs owns a 256-token unit; CTA r holds tokens
// 128 r .. 128 r + 127 and rows [r g/2, r g/2 + g/2) of every tile, and the
// leader's MMA thread issues M = 256 cta_group::2 MMAs whose accumulator lands
// in both CTAs' TMEM.  Otherwise each CTA owns a 128-token unit.
template <int G, bool kPair>
__global__ void __launch_bounds__(kSqThreads, 1) k_sq(const __grid_constant__ SqParams P) {
  using C = Sq<G, kPair>;
  extern __shared__ uint8_t sq_smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[C::kStages];
  __shared__ __align__(8) uint64_t empty_bar[C::kStages];
  __shared__ __align__(8) uint64_t afull_bar[kSqAccBufs];
  __shared__ __align__(8) uint64_t aempty_bar[kSqAccBufs];
  __shared__ __align__(8) uint64_t drain_bar;
  __shared__ uint32_t tmem_base_s;
  __shared__ int abort_s;
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(sq_smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = kPair ? cluster_ctarank() : 0u;   // 0: leader (issues the pair's MMAs)
  uint2* ibuf = reinterpret_cast<uint2*>(smem + C::kStages * C::kStageBytes) + (warp < 2 ? warp : 0) * 32;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int b = 0; b < kSqAccBufs; ++b) {
      mbar_init(&afull_bar[b], 1);
      mbar_init(&aempty_bar[b], (kPair ? 2 : 1) * kSqEpiWarps);   // the epilogue warps of the unit's CTAs
    }
    mbar_init(&drain_bar, 1);
    abort_s = 0;
    fence_mbar_init();
    for (int l = 0; l < P.n_layers; ++l) {
      prefetch_tmap(&P.L[l].xmap);
      for (int h = 0; h < C::R; ++h) prefetch_tmap(&P.L[l].wmap[h]);
    }
  }
  if (warp == 1) {
    if constexpr (kPair) {
      tmem_alloc_pair(&tmem_base_s, kSqTmemCols);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(&tmem_base_s, kSqTmemCols);
      tmem_relinquish();
    }
  }
  tc_fence_before();
  if constexpr (kPair) cluster_sync_all();
  else __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  volatile int* abort_flag = &abort_s;
  const int n_tiles = P.n_tiles;
  const int owner = kPair ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;   // unit owners: CTA pairs or single CTAs
  const int n_owners = kPair ? (int)(gridDim.x >> 1) : (int)gridDim.x;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    uint32_t stage = 0, phase = 0;
    uint32_t armed = 0u, armed_par = 0u;
    bool ok = true;
    for (int kt = 0, t; ok && (t = owner_tile(P.tl, n_tiles, owner, n_owners, kt)) >= 0; ++kt) {
      const SqLayer& L = P.L[sq_layer_of(P, t)];
      const int lt = t - L.tile_begin;
      const int m = lt % L.n_m, w = lt / L.n_m;
      const int tok0 = m * C::kTile + (int)rank * kSqM;
      for (int c0 = 0; c0 < L.Gin && ok; c0 += 32) {
        const int n_it = sq_items(L, w, c0, lane, ibuf);
        if (lane == 0) {
          for (int it = 0; it < n_it && ok; ++it) {
            const uint2 e = ibuf[it];
            const int v = (int)(e.x & 0xFFFFu), n = (int)((e.x >> 16) & 0xFFu), p0 = (int)e.y;
            if (!mbar_wait_bounded(&empty_bar[stage], phase ^ 1u, abort_flag, P.err, kSqWaitLimitNs, kDevErrTimeout)) {
              ok = false;
              break;
            }
            uint8_t* sx = smem + stage * C::kStageBytes;
            if constexpr (kPair) {
              // both CTAs' copies complete on the leader's full barrier, which
              // expects the bytes of both
              if (rank == 0)
                mbar_arrive_expect_tx(&full_bar[stage],
                                      (uint32_t)(2 * P.x_rows * 2 * G) + (uint32_t)(n * G * 2 * G));
              const uint32_t fb = mapa_shared(smem_u32(&full_bar[stage]), 0);
              if constexpr (G > 64) {
                tma_load_3d_pair(sx, &L.xmap, fb, 0, tok0, 2 * v);
                tma_load_3d_pair(sx + C::kSlab, &L.xmap, fb, 0, tok0, 2 * v + 1);
                tma_load_5d_pair(sx + C::kRegion, &L.wmap[0], fb, 0, 0, 0, (int)rank, p0);
              } else {
                tma_load_2d_pair(sx, &L.xmap, fb, v * G, tok0);
                tma_load_4d_pair(sx + C::kRegion, &L.wmap[n - 1], fb, 0, 0, (int)rank, p0);
              }
            } else {
              mbar_arrive_expect_tx(&full_bar[stage], (uint32_t)(P.x_rows * 2 * G) + (uint32_t)(n * G * 2 * G));
              if constexpr (G > 64) {
                // one box per 64-column slab, each into its own slab region (a two-slab
                // box of fewer than 128 rows would pack the slabs back to back)
                tma_load_3d(sx, &L.xmap, &full_bar[stage], 0, tok0, 2 * v);
                tma_load_3d(sx + C::kSlab, &L.xmap, &full_bar[stage], 0, tok0, 2 * v + 1);
                tma_load_3d(sx + C::kRegion, &L.wmap[0], &full_bar[stage], 0, p0 * G, 0);
              } else {
                tma_load_2d(sx, &L.xmap, &full_bar[stage], v * G, tok0);
                tma_load_2d(sx + C::kRegion, &L.wmap[n - 1], &full_bar[stage], 0, p0 * G);
              }
            }
            armed |= 1u << stage;
            armed_par = (armed_par & ~(1u << stage)) | (phase << stage);
            if (++stage == (uint32_t)C::kStages) {
              stage = 0;
              phase ^= 1u;
            }
          }
        }
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      }
    }
    if (lane == 0 && !ok && rank == 0) {
      // let copies already in flight land before the CTA retires
      for (int s = 0; s < C::kStages; ++s) {
        if (!((armed >> s) & 1u)) continue;
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait(&full_bar[s], (armed_par >> s) & 1u))
          if (globaltimer_ns() - t0 > kSqDrainLimitNs) break;
      }
    }
    __syncwarp();
  } else if (warp == 1 && rank == 0) {
    // ------------------------------------------------------------ MMA issuer (leader)
    uint32_t stage = 0, phase = 0;
    int buf = 0;
    uint32_t ae_ph = 0u;
    bool ok = true;
    constexpr uint32_t idesc = idesc_bf16_f32(kPair ? 2 * kSqM : kSqM, G);
    constexpr int kTileRows = kPair ? G / 2 : G;   // rows of each tile this CTA holds
    for (int kt = 0, t; ok && (t = owner_tile(P.tl, n_tiles, owner, n_owners, kt)) >= 0; ++kt) {
      const SqLayer& L = P.L[sq_layer_of(P, t)];
      const int w = (t - L.tile_begin) / L.n_m;
      if (lane == 0) {
        const uint32_t par = ((ae_ph >> buf) & 1u) ^ 1u;
        ok = kPair ? mbar_wait_bounded_cluster(&aempty_bar[buf], par, abort_flag, P.err, kSqWaitLimitNs, kDevErrTimeout)
                   : mbar_wait_bounded(&aempty_bar[buf], par, abort_flag, P.err, kSqWaitLimitNs, kDevErrTimeout);
        ae_ph ^= 1u << buf;
        tc_fence_after();
      }
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      const uint32_t d0 = tmem + (uint32_t)(buf * kSqWin);
      uint32_t seen = 0u;   // block rows of this unit whose accumulator slice holds a result
      for (int c0 = 0; c0 < L.Gin && ok; c0 += 32) {
        const int n_it = sq_items(L, w, c0, lane, ibuf);
        if (lane == 0) {
          for (int it = 0; it < n_it && ok; ++it) {
            const uint32_t mk = ibuf[it].x >> 24;
            if (!mbar_wait_bounded(&full_bar[stage], phase, abort_flag, P.err, kSqWaitLimitNs, kDevErrTimeout)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t sx = smem_u32(smem + stage * C::kStageBytes);
            int i = 0;
#pragma unroll
            for (int b = 0; b < C::R; ++b) {
              if (!((mk >> b) & 1u)) continue;
              const uint32_t d = d0 + (uint32_t)(b * G);
#pragma unroll
              for (int kk = 0; kk < C::kKSteps; ++kk) {
                const uint32_t ka = (uint32_t)((kk >> 2) * C::kSlab + (kk & 3) * 32);
                const uint32_t kb = (uint32_t)((kk >> 2) * C::kWSlab + (kk & 3) * 32);
                const uint64_t ad = sq_desc(sx + ka, C::kSBO, C::kSwz);
                const uint64_t bd =
                    sq_desc(sx + C::kRegion + (uint32_t)(i * kTileRows * C::kRowB) + kb, C::kSBO, C::kSwz);
                const uint32_t acc = (((seen >> b) & 1u) | (uint32_t)kk) != 0u ? 1u : 0u;
                if constexpr (kPair) mma_bf16_ss_pair(d, ad, bd, idesc, acc);
                else mma_bf16_ss(d, ad, bd, idesc, acc);
              }
              seen |= 1u << b;
              ++i;
            }
            if constexpr (kPair) mma_commit_pair_mc(&empty_bar[stage], 0x3);
            else mma_commit(&empty_bar[stage]);
            if (++stage == (uint32_t)C::kStages) {
              stage = 0;
              phase ^= 1u;
            }
          }
        }
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      }
      if (!ok) break;
      // the unit's accumulator is complete once its MMAs are
      if (lane == 0) {
        if constexpr (kPair) mma_commit_pair_mc(&afull_bar[buf], 0x3);
        else mma_commit(&afull_bar[buf]);
      }
      buf ^= 1;
    }
    if (lane == 0) {
      if constexpr (kPair) mma_commit_pair(&drain_bar);
      else mma_commit(&drain_bar);
      mbar_wait_bounded(&drain_bar, 0u, nullptr, P.err, kSqWaitLimitNs, kDevErrTimeout);
    }
    __syncwarp();
  } else if (warp >= 2) {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;   // TMEM lane quarter this warp may access
    int buf = 0;
    uint32_t af_ph = 0u;
    bool ok = true;
    for (int kt = 0, t; ok && (t = owner_tile(P.tl, n_tiles, owner, n_owners, kt)) >= 0; ++kt) {
      const SqLayer& L = P.L[sq_layer_of(P, t)];
      const int lt = t - L.tile_begin;
      const int m = lt % L.n_m, w = lt / L.n_m;
      // block rows with at least one kept tile in the unit (the others are zero)
      uint32_t seen = 0u;
      for (int v = lane; v < L.Gin; v += 32) seen |= L.gwmask[(int64_t)v * L.nwin + w];
      seen = __reduce_or_sync(0xffffffffu, seen);
      if (!mbar_wait_bounded(&afull_bar[buf], (af_ph >> buf) & 1u, abort_flag, P.err, kSqWaitLimitNs,
                             kDevErrTimeout)) {
        ok = false;
        break;
      }
      af_ph ^= 1u << buf;
      tc_fence_after();
      const int tok = m * C::kTile + (int)rank * kSqM + 32 * q + lane;
      uint16_t* yrow = L.y + (int64_t)tok * L.out;
#pragma unroll 1
      for (int j = 0; j < kSqWin / 32; ++j) {
        uint32_t v[32];
        tmem_ld_x32(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * kSqWin + 32 * j), v);
        tmem_wait_ld();
        reg_fence(v);
        const int r0 = w * kSqWin + 32 * j;
        if (tok < P.T) {
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const int rb = r0 + 8 * k;
            const bool keep = (seen >> ((32 * j + 8 * k) / G)) & 1u;
            if (rb + 8 <= L.out) {
              const float* f = reinterpret_cast<const float*>(v + 8 * k);
              *reinterpret_cast<uint4*>(yrow + rb) =
                  make_uint4(sq_pack_bf16x2(f[0], f[1], keep), sq_pack_bf16x2(f[2], f[3], keep),
                             sq_pack_bf16x2(f[4], f[5], keep), sq_pack_bf16x2(f[6], f[7], keep));
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if constexpr (kPair) mbar_arrive_cluster_relaxed(mapa_shared(smem_u32(&aempty_bar[buf]), 0));
        else mbar_arrive(&aempty_bar[buf]);
      }
      buf ^= 1;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (abort_s) {
    // a role gave up: give copies the peer may still have in flight time to land
    const uint64_t t0 = globaltimer_ns();
    while (globaltimer_ns() - t0 < 2000000ull) {
    }
  }
  if constexpr (kPair) cluster_sync_all();
  if (warp == 1) {
    tc_fence_after();
    if constexpr (kPair) tmem_dealloc_pair(tmem, kSqTmemCols);
    else tmem_dealloc(tmem, kSqTmemCols);
  }
  if constexpr (kPair) cluster_sync_all();
}

// ------------------------------------------------------------------ packing
// count: gwmask[v][w] = kept block rows of window w in column block v
__global__ void k_sq_count(const uint8_t* __restrict__ mask, int32_t Gout, int32_t Gin, int32_t R, int32_t nwin,
                           uint8_t* __restrict__ gwmask, int32_t* __restrict__ cnt) {
  const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;   // e = v * nwin + w
  if (e >= (int64_t)Gin * nwin) return;
  const int v = (int)(e / nwin), w = (int)(e % nwin);
  uint32_t bits = 0;
  for (int i = 0; i < R; ++i) {
    const int u = w * R + i;
    if (u < Gout && mask[(int64_t)u * Gin + v] != 0) bits |= 1u << i;
  }
  gwmask[e] = (uint8_t)bits;
  cnt[e] = __popc(bits);
}

__device__ __forceinline__ uint4 sq_ld16(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}

// compact + copy: one warp per group (u, v); a kept group's g x g block is
// copied to its tile (16 bytes per lane per step) and its block row recorded
__global__ void k_sq_compact(const uint16_t* __restrict__ W, const uint8_t* __restrict__ mask, int32_t g,
                             int32_t in, int32_t Gout, int32_t Gin, int32_t R, int32_t nwin,
                             const int32_t* __restrict__ gwoff, const uint8_t* __restrict__ gwmask,
                             int32_t* __restrict__ row_idx, uint16_t* __restrict__ tiles,
                             int32_t* __restrict__ gtidx) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
  const int per_row = g / 8;   // 16-byte pieces per block row
  for (int64_t e = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); e < (int64_t)Gout * Gin;
       e += warps) {
    const int u = (int)(e / Gin), v = (int)(e % Gin);
    if (mask[e] == 0) {
      if (lane == 0) gtidx[e] = -1;
      continue;
    }
    const int w = u / R, i = u % R;
    const uint32_t mk = gwmask[(int64_t)v * nwin + w];
    const int64_t j = gwoff[(int64_t)v * (nwin + 1) + w] + __popc(mk & ((1u << i) - 1u));
    if (lane == 0) gtidx[e] = (int32_t)j;
    uint16_t* dst = tiles + j * (int64_t)g * g;
    for (int c = lane; c < g * per_row; c += 32) {
      const int r = c / per_row, k8 = c % per_row;
      reinterpret_cast<uint4*>(dst + (int64_t)r * g)[k8] =
          sq_ld16(W + ((int64_t)g * u + r) * in + (int64_t)g * v + 8 * k8);
    }
    if (lane == 0) row_idx[j] = u;
  }
}

// unpack: one warp per group; kept groups copied back, pruned groups +0.0
__global__ void k_sq_unpack(const uint16_t* __restrict__ tiles, int32_t g, int32_t in, int32_t Gout, int32_t Gin, int32_t R, int32_t nwin,
                            const int32_t* __restrict__ gwoff, const uint8_t* __restrict__ gwmask,
                            uint16_t* __restrict__ W_hat) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
  const int per_row = g / 8;
  for (int64_t e = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); e < (int64_t)Gout * Gin;
       e += warps) {
    const int u = (int)(e / Gin), v = (int)(e % Gin);
    const int w = u / R, i = u % R;
    const uint32_t mk = gwmask[(int64_t)v * nwin + w];
    const bool kept = (mk >> i) & 1u;
    const int64_t j = gwoff[(int64_t)v * (nwin + 1) + w] + __popc(mk & ((1u << i) - 1u));
    const uint16_t* src = tiles + j * (int64_t)g * g;
    for (int c = lane; c < g * per_row; c += 32) {
      const int r = c / per_row, k8 = c % per_row;
      const uint4 val = kept ? sq_ld16(src + (int64_t)r * g + 8 * k8) : make_uint4(0u, 0u, 0u, 0u);
      reinterpret_cast<uint4*>(W_hat + ((int64_t)g * u + r) * in + (int64_t)g * v)[k8] = val;
    }
  }
}

int sq_grid_for(int64_t warps_needed) {
  int64_t b = (warps_needed + 7) / 8;
  if (b < 1) b = 1;
  if (b > (1 << 20)) b = 1 << 20;
  return (int)b;
}

int sq_sm_count() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 148;
  }
  return n;
}

template <int G, bool kPair>
cudaError_t sq_set_attr() {
  static std::once_flag once;
  static cudaError_t err = cudaSuccess;
  std::call_once(once, []() {
    err = cudaFuncSetAttribute(k_sq<G, kPair>, cudaFuncAttributeMaxDynamicSharedMemorySize, Sq<G, kPair>::kSmem);
  });
  return err;
}

// Above 128 tokens, CTA pairs own 256-token units; up to 128, single CTAs own
// 128-token units (a pair unit would be half empty).
template <int G, bool kPair>
gs_status sq_launch(const void* const* xs, const gs_packed* const* ps, const int* idx, int nb, int64_t T,
                    void* const* ys, int* err, cudaStream_t s) {
  using C = Sq<G, kPair>;
  if (sq_set_attr<G, kPair>() != cudaSuccess) return GS_ERR_CUDA;
  SqParams P;
  std::memset(&P, 0, sizeof(P));
  int64_t tiles = 0;
  const uint32_t xr = (uint32_t)std::min<int64_t>(T, kSqM);
  for (int k = 0; k < nb; ++k) {
    const gs_packed* p = ps[idx[k]];
    SqLayer& L = P.L[k];
    bool ok;
    if (G > 64)
      ok = encode_tmap_slabs_bf16(&L.xmap, xs[idx[k]], (uint64_t)p->in, (uint64_t)T, xr, 1);
    else
      ok = encode_tmap_2d_bf16_swz(&L.xmap, xs[idx[k]], (uint64_t)p->in, (uint64_t)T, G, xr, C::kRowB);
    if (!ok) return GS_ERR_CUDA;
    for (int h = 0; h < C::R; ++h) std::memcpy(&L.wmap[h], kPair ? p->hmaps[h] : p->gmaps[h], sizeof(CUtensorMap));
    L.gwoff = p->gwoff;
    L.gwmask = p->gwmask;
    L.y = static_cast<uint16_t*>(ys[idx[k]]);
    L.out = (int32_t)p->out;
    L.Gin = p->G;
    L.nwin = p->nwin;
    L.n_m = (int32_t)((T + C::kTile - 1) / C::kTile);
    L.tile_begin = (int32_t)tiles;
    tiles += (int64_t)L.n_m * L.nwin;
  }
  if (tiles > INT32_MAX) return GS_ERR_UNSUPPORTED;
  P.n_layers = nb;
  P.T = (int32_t)T;
  P.n_tiles = (int32_t)tiles;
  P.x_rows = (int32_t)xr;
  P.err = err;
  const int owners = (int)std::min<int64_t>(tiles, kPair ? sq_sm_count() / 2 : sq_sm_count());
  if (tiles <= kTileListMax) {
    // a tile's time follows the kept tiles of its window: the layer's mean
    std::vector<int32_t> cost((size_t)tiles);
    for (int k = 0; k < nb; ++k) {
      const gs_packed* p = ps[idx[k]];
      const int32_t c = (int32_t)((p->kept + p->nwin - 1) / std::max<int64_t>(p->nwin, 1));
      for (int64_t t = 0; t < (int64_t)P.L[k].n_m * P.L[k].nwin; ++t) cost[(size_t)(P.L[k].tile_begin + t)] = c;
    }
    plan_tiles(cost, owners, P.tl);
  }
  cudaError_t e;
  if constexpr (kPair) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(2 * owners));
    cfg.blockDim = dim3(kSqThreads);
    cfg.dynamicSmemBytes = C::kSmem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, k_sq<G, true>, P);
  } else {
    k_sq<G, false><<<owners, kSqThreads, C::kSmem, s>>>(P);
    e = cudaGetLastError();
  }
  note_launch();
  return e == cudaSuccess ? GS_OK : GS_ERR_CUDA;
}

template <int G>
gs_status sq_launch_any(const void* const* xs, const gs_packed* const* ps, const int* idx, int nb, int64_t T,
                        void* const* ys, int* err, cudaStream_t s) {
  return T > kSqM ? sq_launch<G, true>(xs, ps, idx, nb, T, ys, err, s)
                  : sq_launch<G, false>(xs, ps, idx, nb, T, ys, err, s);
}

}  // namespace

bool sq_shape_supported(int g_out, int g_in) {
  return g_out == g_in && (g_out == 16 || g_out == 32 || g_out == 64 || g_out == 128);
}

gs_status sq_pack(const void* W, const uint8_t* mask, gs_packed* p, cudaStream_t s) {
  const int g = p->g_out;
  const int R = kSqWin / g;
  const int64_t Gin = p->G, Gout = p->Gout, nwin = p->nwin;
  const int64_t E = Gin * nwin;
  size_t total = 0;
  auto alloc = [&](void** ptr, size_t bytes) -> gs_status {
    if (bytes == 0) {
      *ptr = nullptr;
      return GS_OK;
    }
    const gs_status st = lib_malloc(ptr, bytes);
    if (st == GS_OK) total += bytes;
    return st;
  };
  gs_status st;
  int32_t* cnt = nullptr;
  if ((st = alloc((void**)&p->offsets, sizeof(int64_t) * (size_t)(Gin + 1))) != GS_OK) return st;
  if ((st = alloc((void**)&p->gwoff, sizeof(int32_t) * (size_t)(Gin * (nwin + 1)))) != GS_OK) return st;
  if ((st = alloc((void**)&p->gwmask, (size_t)E)) != GS_OK) return st;
  if ((st = lib_malloc((void**)&cnt, sizeof(int32_t) * (size_t)E)) != GS_OK) return st;
  k_sq_count<<<(unsigned)((E + 255) / 256), 256, 0, s>>>(mask, (int32_t)Gout, (int32_t)Gin, R, (int32_t)nwin,
                                                         p->gwmask, cnt);
  note_launch();
  st = cudaGetLastError() == cudaSuccess ? GS_OK : GS_ERR_CUDA;
  if (st == GS_OK) st = launch_scan_counts(cnt, (int32_t)Gin, (int32_t)nwin, p->gwoff, p->offsets, s);
  int64_t kept = 0;
  if (st == GS_OK && (cudaMemcpyAsync(&kept, p->offsets + Gin, sizeof(int64_t), cudaMemcpyDeviceToHost, s) !=
                          cudaSuccess ||
                      cudaStreamSynchronize(s) != cudaSuccess))
    st = GS_ERR_CUDA;
  cudaFree(cnt);
  if (st != GS_OK) return st;
  p->kept = kept;
  const size_t tile_elems = (size_t)g * (size_t)g;
  if ((st = alloc((void**)&p->row_idx, sizeof(int32_t) * (size_t)kept)) != GS_OK) return st;
  if ((st = alloc((void**)&p->tiles, 2 * tile_elems * (size_t)kept)) != GS_OK) return st;
  if ((st = alloc((void**)&p->gtidx, sizeof(int32_t) * (size_t)(Gout * Gin))) != GS_OK) return st;
  p->device_bytes = total;
  if (kept > 0) {
    k_sq_compact<<<sq_grid_for(Gout * Gin), 256, 0, s>>>(static_cast<const uint16_t*>(W), mask, g, (int32_t)p->in,
                                                         (int32_t)Gout, (int32_t)Gin, R, (int32_t)nwin, p->gwoff,
                                                         p->gwmask, p->row_idx, p->tiles, p->gtidx);
    note_launch();
    if (cudaGetLastError() != cudaSuccess) return GS_ERR_CUDA;
    // W slice descriptors: the tiles as a [K g][g] matrix (g = 128: 64-wide slabs)
    for (int h = 0; h < R; ++h) {
      CUtensorMap m;
      const bool ok = g > 64 ? encode_tmap_slabs_bf16(&m, p->tiles, (uint64_t)g, (uint64_t)kept * g, (uint32_t)g, 2)
                             : encode_tmap_2d_bf16_swz(&m, p->tiles, (uint64_t)g, (uint64_t)kept * g, (uint32_t)g,
                                                       (uint32_t)((h + 1) * g), g >= 64 ? 128 : 2 * g);
      if (!ok) return GS_ERR_CUDA;
      std::memcpy(p->gmaps[h], &m, sizeof(m));
      // CTA-pair halves: the tiles as [K][2 halves][g/2 rows][g] (g = 128: each row as
      // two 64-wide slabs); a box takes one half of 1..8 consecutive tiles
      const uint64_t gg = (uint64_t)g;
      bool okh;
      if (g > 64) {
        const uint64_t dims[5] = {64, gg / 2, 2, 2, (uint64_t)kept};
        const uint64_t str[4] = {2 * gg, 128, gg * gg, 2 * gg * gg};
        const uint32_t box[5] = {64, (uint32_t)(g / 2), 2, 1, 1};
        okh = encode_tmap_nd_bf16(&m, p->tiles, 5, dims, str, box, 128);
      } else {
        const uint64_t dims[4] = {gg, gg / 2, 2, (uint64_t)kept};
        const uint64_t str[3] = {2 * gg, gg * gg, 2 * gg * gg};
        const uint32_t box[4] = {(uint32_t)g, (uint32_t)(g / 2), 1, (uint32_t)(h + 1)};
        okh = encode_tmap_nd_bf16(&m, p->tiles, 4, dims, str, box, g >= 64 ? 128 : 2 * g);
      }
      if (!okh) return GS_ERR_CUDA;
      std::memcpy(p->hmaps[h], &m, sizeof(m));
    }
  }
  return GS_OK;
}

gs_status sq_unpack(const gs_packed* p, void* W_hat, cudaStream_t s) {
  const int g = p->g_out;
  k_sq_unpack<<<sq_grid_for((int64_t)p->Gout * p->G), 256, 0, s>>>(
      p->tiles, g, (int32_t)p->in, p->Gout, p->G, kSqWin / g, p->nwin, p->gwoff, p->gwmask,
      static_cast<uint16_t*>(W_hat));
  note_launch();
  return cudaGetLastError() == cudaSuccess ? GS_OK : GS_ERR_CUDA;
}

void sq_release(gs_packed* p) {
  if (p->gwoff) cudaFree(p->gwoff);
  if (p->gwmask) cudaFree(p->gwmask);
  if (p->gtidx) cudaFree(p->gtidx);
  p->gwoff = nullptr;
  p->gwmask = nullptr;
  p->gtidx = nullptr;
}

gs_status sq_linear_batched(const void* const* xs, const gs_packed* const* ps, int n, int64_t T, void* const* ys,
                            cudaStream_t s) {
  if (T <= 0 || n <= 0) return GS_OK;
  int* err = device_error_flag();
  if (!err) return GS_ERR_CUDA;
  // layers without kept groups produce zeros; the others share launches by
  // group size, up to kSqMaxLayers each, most work per unit first
  std::vector<int> order[4];
  for (int i = 0; i < n; ++i) {
    const gs_packed* p = ps[i];
    if (p->kept == 0) {
      if (cudaMemsetAsync(ys[i], 0, (size_t)T * (size_t)p->out * 2, s) != cudaSuccess) return GS_ERR_CUDA;
      continue;
    }
    const int gi = p->g_out == 16 ? 0 : p->g_out == 32 ? 1 : p->g_out == 64 ? 2 : 3;
    order[gi].push_back(i);
  }
  for (int gi = 0; gi < 4; ++gi) {
    std::vector<int>& o = order[gi];
    std::stable_sort(o.begin(), o.end(), [&](int a, int b) {
      return (double)ps[a]->kept / ps[a]->nwin > (double)ps[b]->kept / ps[b]->nwin;
    });
    // Per layer, by its group size, input width and T only (so a batched call
    // gives each layer what a single call gives it):
    //  - decode regime: the tile-streaming kernel, one launch per 16 tokens.  Its
    //    time grows with the 16-token blocks while the tensor-core kernels' stays
    //    flat up to 128 tokens.  Over the five LLaMA-2 7B / 13B projection shapes
    //    at d = 0.5 the zero-filled-window kernel (layers whose input is whole
    //    128-column items, g <= 64) takes 1.3-1.5x its time at 32 tokens,
    //    0.90-1.03x at 48 and 0.37-0.43x at 128; the square tensor-core kernel
    //    (the other layers) breaks even at 128 / 64 / 32 / 16 tokens for
    //    g = 16 / 32 / 64 / 128;
    //  - above it, the zero-filled-window kernel where it applies (dense-layer
    //    tensor work, no per-column-block handshake: the faster of the two at
    //    small tiles), else the square tensor-core kernel.
    const int g = 16 << gi;
    std::vector<int> dec, dense, rest;
    for (int i : o) {
      const bool zf = g <= kSqDenseMaxG && ps[i]->in % 128 == 0;
      (T <= (zf ? (int64_t)kSqDecodeMaxTokensZf : (int64_t)(2048 / g)) ? dec : zf ? dense : rest).push_back(i);
    }
    if (!dec.empty()) {
      std::stable_sort(dec.begin(), dec.end(), [&](int a, int b) { return ps[a]->in > ps[b]->in; });   // heaviest rows first
      const int blk = sq_decode_max_tokens();
      std::vector<const void*> xb(n);
      std::vector<void*> yb(n);
      for (int64_t t0 = 0; t0 < T; t0 += blk) {
        const int tb = (int)std::min<int64_t>(blk, T - t0);
        for (int i : dec) {
          xb[i] = static_cast<const uint16_t*>(xs[i]) + t0 * ps[i]->in;
          yb[i] = static_cast<uint16_t*>(ys[i]) + t0 * ps[i]->out;
        }
        for (size_t b0 = 0; b0 < dec.size(); b0 += kSqMaxLayers) {
          const int nb = (int)std::min<size_t>(kSqMaxLayers, dec.size() - b0);
          const gs_status st = sq_decode_batched(xb.data(), ps, dec.data() + b0, nb, tb, yb.data(), s);
          if (st != GS_OK) return st;
        }
      }
    }
    if (!dense.empty()) {
      const gs_status st = launch_prefill_dense(xs, ps, (int)dense.size(), T, ys, s, dense.data());
      if (st != GS_OK) return st;
    }
    o = rest;
    for (size_t b0 = 0; b0 < o.size(); b0 += kSqMaxLayers) {
      const int nb = (int)std::min<size_t>(kSqMaxLayers, o.size() - b0);
      gs_status st;
      switch (gi) {
        case 0: st = sq_launch_any<16>(xs, ps, o.data() + b0, nb, T, ys, err, s); break;
        case 1: st = sq_launch_any<32>(xs, ps, o.data() + b0, nb, T, ys, err, s); break;
        case 2: st = sq_launch_any<64>(xs, ps, o.data() + b0, nb, T, ys, err, s); break;
        default: st = sq_launch_any<128>(xs, ps, o.data() + b0, nb, T, ys, err, s); break;
      }
      if (st != GS_OK) return st;
    }
  }
  return GS_OK;
}

}  // namespace gs
