// Prefill-regime group-sparse linear (many tokens, tensor-core bound):
//   y[t, r] = sum over kept groups (r, c) of X_c[t, :] . W[r, 256c : 256c+256]   (Eq. 1)
//
// Tiles.  A tile is a token range x 160 output rows (a "window").  For every
// chunk c the kept rows of the window form one contiguous slice of the packed
// tiles (rows are ascending inside a chunk), so the slice is a dense K-major
// operand that TMA loads as-is.  Per chunk one tcgen05 MMA chain computes
// D[tokens x n] = X_c . W_slice^T (n <= 160 kept rows, rounded up to 16) into
// one of three TMEM scratch buffers; the epilogue warps then add each window
// row's scratch column (a zero column for rows pruned in chunk c) into the
// window accumulator, which they hold in registers.  W (.) M is never
// materialised and pruned groups cost neither bytes nor FLOPs.
//
// Tile owners.  Normally a CTA pair (a cluster of two CTAs) owns a 256-token
// tile: CTA r holds tokens 128r..128r+127 and half of each W slice, and the
// leader's MMA thread issues M = 256 cta_group::2 MMAs whose D lands in both
// CTAs' TMEM.  Up to 128 tokens (a pair tile would be half empty) each CTA
// owns a 128-token tile, loads whole slices and issues its own M = 128 MMAs.
// One launch walks the tiles of up to kMaxLayers layers that share T.
//
// Copies: a pipeline stage carries 128 of the chunk's 256 k as two 64-wide
// slabs, fetched with one 3-D TMA box for X (128 rows x 2 slabs) and one for
// the W slice (half or whole, from a descriptor with that box height).
// TMA issue costs a fixed ~60-120 cycles per box whatever its size, so two
// large boxes per stage keep the producer far below the copy time.
//
// Roles (one CTA per SM, tile owners persistent over tiles):
//   warp 0      TMA producer
//   warp 1      TMEM allocator + single-thread MMA issuer
//   warps 2..17 epilogue: warp (q, g) owns tokens 32q..32q+31 (its TMEM lane
//               quarter) and window rows 40g..40g+39: 40 fp32 accumulators
//               per thread, updated from 40 single-column TMEM loads per chunk
//               (pruned rows read a zero column) with one wait, then written
//               to y as bf16 at the end of the tile.
// Each warp stages the window's per-chunk slice bounds in shared memory at the
// start of a tile; the epilogue prefetches its blocks' masks four chunks ahead.
// Every mbarrier wait is bounded; a wait that runs out raises a CTA-wide abort
// flag and the library's device error flag, and all roles wind down.
#include "gs_common.cuh"
#include "gs_sm100.cuh"

#include <cuda.h>
#include <algorithm>
#include <cstring>
#include <vector>
#include <mutex>

namespace gs {
namespace {
using namespace sm100;

constexpr int kBM = 128;                      // tokens per CTA (TMEM lanes); a CTA pair covers 256
constexpr int kPairM = 2 * kBM;               // tokens per pair tile
constexpr int kFW = 160;                      // output rows per tile (a window)
constexpr int kGroups = 4;                    // epilogue warps per TMEM lane quarter
constexpr int kRowsPerWarp = kFW / kGroups;   // 40 window rows per epilogue warp
constexpr int kBlkRows = kWin16;              // rows per kept-mask block
constexpr int kMetaBlocks = 3;                // 16-row blocks a warp's 40 rows can touch
constexpr int kNMax = kFW;                    // kept rows per MMA item: a whole window's slice always fits
constexpr int kNMaps = kNMax / 16;            // W descriptors, box heights 8, 16, ..., 80 (half a slice each)
constexpr int kBK = 64;                       // k per slab: one 128-byte swizzle row
constexpr int kSlabs = 2;                     // slabs per pipeline stage (a stage carries 128 k)
constexpr int kStages = 4;
constexpr int kXSlabBytes = kBM * kBK * 2;    // 16 KB
constexpr int kXStageBytes = kSlabs * kXSlabBytes;
constexpr int kWStageBytes = kSlabs * (kNMax / 2) * kBK * 2;   // 20 KB: this CTA's half of the largest slice
constexpr int kStageBytes = kXStageBytes + kWStageBytes;       // 52 KB
constexpr int kScrBufs = 3;                   // TMEM scratch buffers (MMA runs up to two chunks ahead)
constexpr int kEpiWarps = 4 * kGroups;
constexpr int kWarps = 2 + kEpiWarps;
constexpr int kThreads = kWarps * 32;
constexpr int kMaxG = 256;                    // chunks per layer handled by this kernel (in <= 65536)
constexpr int kMetaInts = 2 * kMaxG;          // producer / MMA warp: a tile's item list (int2 per chunk)
constexpr uint32_t kTmemCols = 512;
constexpr int kAcc = kRowsPerWarp;            // 40 accumulators per epilogue thread
constexpr uint32_t kZeroCol = kScrBufs * kNMax;   // 32 columns held at 0.0: the gather source of pruned rows
constexpr int kTblBytes = 2 * kEpiWarps * kAcc * 4;   // per epilogue warp, two chunks: the TMEM address of each row
constexpr uint64_t kWaitLimitNs = 2000000000ull;
constexpr uint64_t kDrainLimitNs = 200000000ull;
constexpr int kSmemBytes = kStages * kStageBytes + 2 * kMetaInts * 4 + kTblBytes + 1024;

// Single-CTA tiles (T <= 128, where a pair tile would be half empty): each CTA
// loads its tile's whole slice per stage and issues its own M = 128 MMAs.
constexpr int kWStageBytesSingle = kSlabs * kNMax * kBK * 2;          // 40 KB: a whole slice
constexpr int kStageBytesSingle = kXStageBytes + kWStageBytesSingle;  // 72 KB
constexpr int kStagesSingle = 3;
constexpr int kSmemBytesSingle = kStagesSingle * kStageBytesSingle + 2 * kMetaInts * 4 + kTblBytes + 1024;
static_assert(kStagesSingle <= kStages, "barrier arrays are sized for the pair layout");
static_assert(kStageBytesSingle % 1024 == 0, "stages must keep 1024-byte alignment");
static_assert(kSmemBytesSingle <= 227 * 1024, "shared memory budget (single-CTA tiles)");

static_assert(kZeroCol + 32 <= kTmemCols, "TMEM budget (scratch buffers + zero columns)");
static_assert(kStageBytes % 1024 == 0 && kXSlabBytes % 1024 == 0, "stages must keep 1024-byte alignment");
static_assert(kFW % 32 == 0 && kRowsPerWarp % 8 == 0 && kNMax % 16 == 0, "tile shape");
static_assert(kRowsPerWarp <= 32 + 8, "the address table is built in two lane rounds");
static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");

// One launch covers up to kMaxLayers layers with the same T; the pairs walk
// one list of tiles, layer after layer (tile_begin = first tile of a layer).
constexpr int kMaxLayers = 8;
struct PrefillLayer {
  CUtensorMap xmap;          // x as (64, T, in/64) slabs, box 64 x 128 x 2
  CUtensorMap wmap[kNMaps];  // tiles as (64, kept, 4) slabs, box 64 x h(i+1) x 2: h = 8 (pair halves) or 16 (whole slices)
  const int32_t* win_off16;
  const uint16_t* kmask16;
  uint16_t* y;
  int32_t out, G, nw16;
  int32_t n_m, n_w;          // pair tiles: ceil(T / 256) x ceil(out / 160)
  int32_t tile_begin;
};
struct PrefillParams {
  PrefillLayer L[kMaxLayers];
  int32_t n_layers, T, n_tiles;
  int* err;
  uint64_t inject_ns;        // test hook: tile owner 0 first waits this long on a word nothing sets (0 = off)
  TileList tl;               // which owner takes which tiles
};

// layer of global tile t
__device__ __forceinline__ int tile_layer(const PrefillParams& P, int t) {
  int l = 0;
  while (l + 1 < P.n_layers && P.L[l + 1].tile_begin <= t) ++l;
  return l;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// Items of a tile: the chunks whose window slice (kept rows = packed rows
// [p0, p1)) is non-empty, in chunk order.  The warp builds the list in shared
// memory, 32 chunks per round: entry = {chunk | (rows rounded up to 16) << 16, p0}.
__device__ __forceinline__ int load_tile_items(const PrefillLayer& P, int w, int lane, int2* items) {
  const int wlo = (kFW / kWin16) * w;
  const int whi = min(wlo + kFW / kWin16, P.nw16);
  int n = 0;
  for (int c0 = 0; c0 < P.G; c0 += 32) {
    const int c = c0 + lane;
    int p0 = 0, p1 = 0;
    if (c < P.G) {
      const int32_t* wo = P.win_off16 + (int64_t)c * (P.nw16 + 1);
      p0 = wo[wlo];
      p1 = wo[whi];
    }
    const bool nonempty = p1 > p0;
    const uint32_t ballot = __ballot_sync(0xffffffffu, nonempty);
    if (nonempty)
      items[n + __popc(ballot & ((1u << lane) - 1u))] = make_int2(c | (((p1 - p0 + 15) & ~15) << 16), p0);
    n += __popc(ballot);
  }
  __syncwarp();
  return n;
}

// Read-only global loads kept at their place in the program: volatile asm is
// not moved across the other volatile asm (barrier waits, TMEM traffic), so a
// load issued chunks ahead of its use is not sunk down to that use.
__device__ __forceinline__ int ld_pinned_s32(const int32_t* p) {
  int v;
  asm volatile("ld.global.nc.b32 %0, [%1];" : "=r"(v) : "l"(p));
  return v;
}
__device__ __forceinline__ uint32_t ld_pinned_u16(const uint16_t* p) {
  uint16_t v;
  asm volatile("ld.global.nc.b16 %0, [%1];" : "=h"(v) : "l"(p));
  return v;
}

// Chunk c's metadata for an epilogue warp: lanes 0..2 fetch (window offset,
// kept mask) of the 16-row blocks its 40 rows touch (from block wblk0); lanes
// 30 and 31 fetch the window slice's start and end.  Chunks past the last read as empty.
__device__ __forceinline__ void load_chunk_meta(const PrefillLayer& P, int c, int wlo, int whi, int wblk0, int lane,
                                                int& bnd, int& woff, uint32_t& km) {
  bnd = 0;
  woff = 0;
  km = 0u;
  if (c >= P.G) return;
  const int32_t* wo = P.win_off16 + (int64_t)c * (P.nw16 + 1);
  const int wi = wblk0 + lane;
  if (lane < kMetaBlocks && wi < P.nw16) {
    woff = ld_pinned_s32(wo + wi);
    km = ld_pinned_u16(P.kmask16 + (int64_t)c * P.nw16 + wi);
  }
  if (lane == 30) bnd = ld_pinned_s32(wo + wlo);
  if (lane == 31) bnd = ld_pinned_s32(wo + whi);
}

// acc[0..n) += v[0..n), two lanes per packed f32x2 add
template <int N>
__device__ __forceinline__ void add_f32x2(float* acc, const uint32_t* v) {
#pragma unroll
  for (int j = 0; j < N; j += 2)
    asm("{\n\t.reg .b64 a, b;\n\t"
        "mov.b64 a, {%0, %1};\n\t"
        "mov.b64 b, {%2, %3};\n\t"
        "add.rn.f32x2 a, a, b;\n\t"
        "mov.b64 {%0, %1}, a;\n\t}"
        : "+f"(acc[j]), "+f"(acc[j + 1])
        : "r"(v[j]), "r"(v[j + 1]));
}

// Single-column TMEM loads of N rows whose addresses sit in shared memory.
template <int N>
__device__ __forceinline__ void gather_rows(const uint32_t* tbl, uint32_t* v) {
#pragma unroll
  for (int j = 0; j < N; j += 4) {
    const uint4 a = *reinterpret_cast<const uint4*>(tbl + j);
    v[j + 0] = tmem_ld_x1(a.x);
    v[j + 1] = tmem_ld_x1(a.y);
    v[j + 2] = tmem_ld_x1(a.z);
    v[j + 3] = tmem_ld_x1(a.w);
  }
}

// KW = chunk width: 256 (1 x 256 groups, two stages per chunk) or 128 (1 x 128 groups, one stage)
template <bool kPair, int KW>
__global__ void __launch_bounds__(kThreads, 1) k_prefill(const __grid_constant__ PrefillParams P) {
  constexpr int kKSteps = KW / (kBK * kSlabs);
  static_assert(KW == 128 || KW == 256, "chunk width");
  constexpr int kStg = kPair ? kStages : kStagesSingle;
  constexpr int kStgBytes = kPair ? kStageBytes : kStageBytesSingle;
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kStages];
  __shared__ __align__(8) uint64_t empty_bar[kStages];
  __shared__ __align__(8) uint64_t sfull_bar[kScrBufs];
  __shared__ __align__(8) uint64_t sempty_bar[kScrBufs];
  __shared__ __align__(8) uint64_t drain_bar;
  __shared__ uint32_t tmem_base_s;
  __shared__ int abort_s;

  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = kPair ? cluster_ctarank() : 0u;   // 0: leader (issues the pair's MMAs), 1: peer
  int2* items = reinterpret_cast<int2*>(smem + kStg * kStgBytes) + (warp < 2 ? warp : 0) * kMaxG;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStg; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int b = 0; b < kScrBufs; ++b) {
      mbar_init(&sfull_bar[b], 1);
      mbar_init(&sempty_bar[b], (kPair ? 2 : 1) * kEpiWarps);   // the epilogue warps of the tile's CTAs
    }
    mbar_init(&drain_bar, 1);
    abort_s = 0;
    fence_mbar_init();
    for (int l = 0; l < P.n_layers; ++l) {
      prefetch_tmap(&P.L[l].xmap);
      for (int h = 0; h < kNMaps; ++h) prefetch_tmap(&P.L[l].wmap[h]);
    }
  }
  if (warp == 1) {
    if constexpr (kPair) {
      tmem_alloc_pair(&tmem_base_s, kTmemCols);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(&tmem_base_s, kTmemCols);
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
  // tile owners: CTA pairs, or single CTAs
  const int pair = kPair ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
  const int n_pairs = kPair ? (int)(gridDim.x >> 1) : (int)gridDim.x;

  if (P.inject_ns != 0 && pair == 0) {
    // test hook: before any copy or MMA is issued, a bounded wait on a word
    // that nothing sets runs out in each CTA of tile owner 0; the owner then
    // records the timeout and skips its tiles (every role, both CTAs)
    if (threadIdx.x == 0) {
      const volatile int* never = P.err + 1;
      const uint64_t t0 = globaltimer_ns();
      while (*never == 0) {
        if (globaltimer_ns() - t0 > P.inject_ns) {
          atomicExch(P.err, kDevErrTimeout);
          abort_s = 1;
          break;
        }
        __nanosleep(1000);
      }
    }
    __syncthreads();
  }
  const bool injected_abort = pair == 0 && abort_s != 0;

  if (injected_abort) {
    // nothing was issued: go straight to the TMEM release
  } else if (warp == 0) {
    // ------------------------------------------------------------ producer
    uint32_t stage = 0, phase = 0;
    uint32_t armed = 0u, armed_par = 0u;   // per stage: a copy was issued / the phase it completes
    bool ok = true;
    for (int kt = 0, t; ok && (t = owner_tile(P.tl, n_tiles, pair, n_pairs, kt)) >= 0; ++kt) {
      const PrefillLayer& L = P.L[tile_layer(P, t)];
      const int lt = t - L.tile_begin;
      const int m = lt % L.n_m, w = lt / L.n_m;
      const int n_items = load_tile_items(L, w, lane, items);
      if (lane == 0) {
        for (int it = 0; it < n_items && ok; ++it) {
          const int2 e = items[it];
          const int c = e.x & 0xFFFF, nr = e.x >> 16, start = e.y;
          const int hn = nr >> 1;   // slice rows held by each CTA of the pair
          const CUtensorMap* wm = kPair ? &L.wmap[(hn >> 3) - 1] : &L.wmap[(nr >> 4) - 1];
          for (int ks = 0; ks < kKSteps; ++ks) {
            if (!mbar_wait_bounded(&empty_bar[stage], phase ^ 1u, abort_flag, P.err, kWaitLimitNs,
                                   kDevErrTimeout)) {
              ok = false;
              break;
            }
            uint8_t* sx = smem + stage * kStgBytes;
            if constexpr (kPair) {
              // both CTAs' copies complete on the leader's full barrier, which
              // expects the bytes of the two halves
              if (rank == 0)
                mbar_arrive_expect_tx(&full_bar[stage], (uint32_t)(2 * kXStageBytes + nr * kSlabs * kBK * 2));
              const uint32_t fb = mapa_shared(smem_u32(&full_bar[stage]), 0);
              tma_load_3d_pair(sx, &L.xmap, fb, 0, m * kPairM + (int)rank * kBM, c * (KW / kBK) + ks * kSlabs);
              tma_load_3d_pair(sx + kXStageBytes, wm, fb, 0, start + (int)rank * hn, ks * kSlabs);
            } else {
              mbar_arrive_expect_tx(&full_bar[stage], (uint32_t)(kXStageBytes + nr * kSlabs * kBK * 2));
              tma_load_3d(sx, &L.xmap, &full_bar[stage], 0, m * kBM, c * (KW / kBK) + ks * kSlabs);
              tma_load_3d(sx + kXStageBytes, wm, &full_bar[stage], 0, start, ks * kSlabs);
            }
            armed |= 1u << stage;
            armed_par = (armed_par & ~(1u << stage)) | (phase << stage);
            if (++stage == kStg) {
              stage = 0;
              phase ^= 1u;
            }
          }
        }
      }
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
    }
    if (lane == 0 && !ok && rank == 0) {
      // let copies already in flight land before the CTA retires
      for (int s = 0; s < kStg; ++s) {
        if (!((armed >> s) & 1u)) continue;
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait(&full_bar[s], (armed_par >> s) & 1u))
          if (globaltimer_ns() - t0 > kDrainLimitNs) break;
      }
    }
    __syncwarp();
  } else if (warp == 1 && rank == 0) {
    // ------------------------------------------------------------ MMA issuer (leader CTA)
    uint32_t stage = 0, phase = 0;
    int buf = 0;
    uint32_t se_ph = 0u;   // bit b: parity of scratch buffer b's next release
    bool ok = true;
    for (int kt = 0, t; ok && (t = owner_tile(P.tl, n_tiles, pair, n_pairs, kt)) >= 0; ++kt) {
      const PrefillLayer& L = P.L[tile_layer(P, t)];
      const int w = (t - L.tile_begin) / L.n_m;
      const int n_items = load_tile_items(L, w, lane, items);
      if (lane == 0) {
        for (int it = 0; it < n_items && ok; ++it) {
          const int nr = items[it].x >> 16;
          const bool freed =
              kPair ? mbar_wait_bounded_cluster(&sempty_bar[buf], ((se_ph >> buf) & 1u) ^ 1u, abort_flag, P.err,
                                                kWaitLimitNs, kDevErrTimeout)
                    : mbar_wait_bounded(&sempty_bar[buf], ((se_ph >> buf) & 1u) ^ 1u, abort_flag, P.err, kWaitLimitNs,
                                        kDevErrTimeout);
          if (!freed) {
            ok = false;
            break;
          }
          se_ph ^= 1u << buf;
          tc_fence_after();
          const uint32_t d = tmem + (uint32_t)(buf * kNMax);
          const uint32_t idesc = idesc_bf16_f32(kPair ? kPairM : kBM, nr);
          for (int ks = 0; ks < kKSteps; ++ks) {
            if (!mbar_wait_bounded(&full_bar[stage], phase, abort_flag, P.err, kWaitLimitNs, kDevErrTimeout)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t sx = smem_u32(smem + stage * kStgBytes);
#pragma unroll
            for (int j = 0; j < kSlabs; ++j) {
              const uint64_t ad = sdesc_sw128(sx + j * kXSlabBytes);
              const uint64_t bd = sdesc_sw128(sx + kXStageBytes + j * (kPair ? (nr >> 1) : nr) * (kBK * 2));
#pragma unroll
              for (int kk = 0; kk < kBK / 16; ++kk) {
                if constexpr (kPair)
                  mma_bf16_ss_pair(d, ad + (uint64_t)(2 * kk), bd + (uint64_t)(2 * kk), idesc,
                                   (ks | j | kk) != 0 ? 1u : 0u);
                else
                  mma_bf16_ss(d, ad + (uint64_t)(2 * kk), bd + (uint64_t)(2 * kk), idesc, (ks | j | kk) != 0 ? 1u : 0u);
              }
            }
            if constexpr (kPair) mma_commit_pair_mc(&empty_bar[stage], 0x3);
            else mma_commit(&empty_bar[stage]);
            if (++stage == kStg) {
              stage = 0;
              phase ^= 1u;
            }
          }
          if (!ok) break;
          if constexpr (kPair) mma_commit_pair_mc(&sfull_bar[buf], 0x3);
          else mma_commit(&sfull_bar[buf]);
          if (++buf == kScrBufs) buf = 0;
        }
      }
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
    }
    if (lane == 0) {
      // all MMAs issued by this thread have completed once drain_bar flips
      if constexpr (kPair) mma_commit_pair(&drain_bar);
      else mma_commit(&drain_bar);
      mbar_wait_bounded(&drain_bar, 0u, nullptr, P.err, kWaitLimitNs, kDevErrTimeout);
    }
    __syncwarp();
  } else if (warp >= 2) {
    // ------------------------------------------------------------ epilogue
    // Warp (q, g): TMEM lane quarter q (tokens 32q..32q+31) and window rows
    // 40g .. 40g+39.
    const int ew = warp - 2;
    const int q = warp & 3;
    const int g = ew >> 2;
    const uint32_t t_scr = tmem + ((uint32_t)(32 * q) << 16);
    const uint32_t t_zero = t_scr + kZeroCol;
    tmem_st_x32_zero(t_zero);
    tmem_wait_st();
    uint32_t* tbl = reinterpret_cast<uint32_t*>(smem + kStg * kStgBytes + 2 * kMetaInts * 4) + ew * 2 * kAcc;
    int buf = 0;
    uint32_t sf_ph = 0u;   // bit b: parity of scratch buffer b's next fill
    bool ok = true;
    for (int kt = 0, t; ok && (t = owner_tile(P.tl, n_tiles, pair, n_pairs, kt)) >= 0; ++kt) {
      const PrefillLayer& L = P.L[tile_layer(P, t)];
      const int lt = t - L.tile_begin;
      const int m = lt % L.n_m, w = lt / L.n_m;
      const int r0 = w * kFW + kRowsPerWarp * g;
      const int wblk0 = (kFW / kWin16) * w + (kRowsPerWarp * g) / kBlkRows;
      const int rsh = (kRowsPerWarp * g) % kBlkRows;   // the warp's first row within block wblk0
      float acc[kAcc];
#pragma unroll
      for (int i = 0; i < kAcc; ++i) acc[i] = 0.f;
      // per chunk: the window's slice bounds and this half's block metadata,
      // prefetched four chunks ahead into four register slots.  The loop is
      // unrolled by four so a slot is read (its load long complete) and only
      // then reloaded; no register copy ever waits on a load in flight.
      const int wlo = (kFW / kWin16) * w, whi = min(wlo + kFW / kWin16, L.nw16);
      int bnd0, bnd1, bnd2, bnd3, wo0, wo1, wo2, wo3;
      uint32_t km0, km1, km2, km3;
      load_chunk_meta(L, 0, wlo, whi, wblk0, lane, bnd0, wo0, km0);
      load_chunk_meta(L, 1, wlo, whi, wblk0, lane, bnd1, wo1, km1);
      load_chunk_meta(L, 2, wlo, whi, wblk0, lane, bnd2, wo2, km2);
      load_chunk_meta(L, 3, wlo, whi, wblk0, lane, bnd3, wo3, km3);
      // Gather addresses of a chunk (its metadata slot), for scratch buffer
      // `buf`: row r of the warp (window row 40g + r: block k, bit i; kept
      // mask m, first kept row at scratch column b0) reads scratch column
      // b0 + popc(m & (2^i - 1)) when kept and a zero column when pruned.
      // The lanes compute the 40 addresses (rows lane, lane + 32).
      auto build_table = [&](uint32_t* t, int bnd, int woff, uint32_t km) {
        const int p0 = __shfl_sync(0xffffffffu, bnd, 30);
        const uint32_t scr = t_scr + (uint32_t)(buf * kNMax);
#pragma unroll
        for (int rr = 0; rr < 2; ++rr) {
          const int r = lane + 32 * rr;
          const int k = (r + rsh) >> 4, i = (r + rsh) & 15;
          const uint32_t mk = __shfl_sync(0xffffffffu, km, k);   // lanes >= 3 hold no block: mask 0
          const int wo = __shfl_sync(0xffffffffu, woff, k);
          const uint32_t addr =
              ((mk >> i) & 1u) ? scr + (uint32_t)(wo - p0 + __popc(mk & ((1u << i) - 1u))) : t_zero;
          if (r < kAcc) t[r] = addr;
        }
        __syncwarp();
      };
      // One chunk.  Its address table was built by the previous step, so the
      // path from "scratch full" to "scratch free" holds only the table reads,
      // the 40 TMEM loads and their wait; the next chunk's table is built
      // after the buffer is handed back, then the loaded values are added.
      auto step = [&](int c, int& bnd, int& wo, uint32_t& kmr, int bnd_n, int wo_n, uint32_t km_n) {
        const int p0 = __shfl_sync(0xffffffffu, bnd, 30), p1 = __shfl_sync(0xffffffffu, bnd, 31);
        load_chunk_meta(L, c + 4, wlo, whi, wblk0, lane, bnd, wo, kmr);
        uint32_t* t_cur = tbl + (c & 1) * kAcc;
        uint32_t* t_next = tbl + ((c + 1) & 1) * kAcc;
        if (p1 <= p0 || !ok) {
          build_table(t_next, bnd_n, wo_n, km_n);
          return;
        }
        if (!mbar_wait_bounded(&sfull_bar[buf], (sf_ph >> buf) & 1u, abort_flag, P.err, kWaitLimitNs,
                               kDevErrTimeout)) {
          ok = false;
          return;
        }
        sf_ph ^= 1u << buf;
        tc_fence_after();
        uint32_t v[kAcc];
        gather_rows<kAcc>(t_cur, v);
        tmem_wait_ld();
        reg_fence(v);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if constexpr (kPair) mbar_arrive_cluster_relaxed(mapa_shared(smem_u32(&sempty_bar[buf]), 0));
          else mbar_arrive(&sempty_bar[buf]);
        }
        if (++buf == kScrBufs) buf = 0;
        build_table(t_next, bnd_n, wo_n, km_n);
        add_f32x2<kAcc>(acc, v);
      };
      build_table(tbl, bnd0, wo0, km0);
      for (int c = 0; c < L.G && ok; c += 4) {
        step(c, bnd0, wo0, km0, bnd1, wo1, km1);
        if (c + 1 < L.G) step(c + 1, bnd1, wo1, km1, bnd2, wo2, km2);
        if (c + 2 < L.G) step(c + 2, bnd2, wo2, km2, bnd3, wo3, km3);
        if (c + 3 < L.G) step(c + 3, bnd3, wo3, km3, bnd0, wo0, km0);
      }
      if (!ok) break;
      // accumulators -> bf16 y rows [r0, r0 + 40) of token tok
      const int tok = (kPair ? m * kPairM + (int)rank * kBM : m * kBM) + 32 * q + lane;
      if (tok < P.T) {
        uint16_t* yrow = L.y + (int64_t)tok * L.out;
        const bool vec_ok = (L.out & 7) == 0;
#pragma unroll
        for (int k = 0; k < kAcc / 8; ++k) {
          const int rb = r0 + 8 * k;
          const float* a = acc + 8 * k;
          if (vec_ok && rb + 8 <= L.out) {
            *reinterpret_cast<uint4*>(yrow + rb) =
                make_uint4(pack_bf16x2(a[0], a[1]), pack_bf16x2(a[2], a[3]), pack_bf16x2(a[4], a[5]),
                           pack_bf16x2(a[6], a[7]));
          } else {
#pragma unroll
            for (int i = 0; i < 8; ++i)
              if (rb + i < L.out) yrow[rb + i] = __bfloat16_as_ushort(__float2bfloat16_rn(a[i]));
          }
        }
      }
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
  else __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    if constexpr (kPair) tmem_dealloc_pair(tmem, kTmemCols);
    else tmem_dealloc(tmem, kTmemCols);
  }
  if constexpr (kPair) cluster_sync_all();
  else __syncthreads();
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
  static_assert(sizeof(p->wmaps) / sizeof(p->wmaps[0]) == kNMaps, "one W descriptor per slice height");
  for (int h = 0; h < kNMaps; ++h) {
    CUtensorMap m;
    if (!encode_tmap_slabs_bf16(&m, p->tiles, (uint64_t)p->g_in, (uint64_t)p->kept, (uint32_t)(8 * (h + 1)), kSlabs))
      return GS_ERR_CUDA;
    std::memcpy(p->wmaps[h], &m, sizeof(m));
    if (!encode_tmap_slabs_bf16(&m, p->tiles, (uint64_t)p->g_in, (uint64_t)p->kept, (uint32_t)(16 * (h + 1)), kSlabs))
      return GS_ERR_CUDA;
    std::memcpy(p->wmaps_full[h], &m, sizeof(m));
  }
  p->wmaps_valid = true;
  return GS_OK;
}

int prefill_max_chunks() { return kMaxG; }

gs_status launch_prefill_batched(const void* const* xs, const gs_packed* const* ps, int n, int64_t T,
                                 void* const* ys, cudaStream_t s) {
  if (T <= 0 || n <= 0) return GS_OK;
  static std::once_flag attr_once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(attr_once, []() {
    attr_err = cudaFuncSetAttribute(k_prefill<true, 256>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
    if (attr_err == cudaSuccess)
      attr_err = cudaFuncSetAttribute(k_prefill<false, 256>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      kSmemBytesSingle);
    if (attr_err == cudaSuccess)
      attr_err = cudaFuncSetAttribute(k_prefill<true, 128>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
    if (attr_err == cudaSuccess)
      attr_err = cudaFuncSetAttribute(k_prefill<false, 128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      kSmemBytesSingle);
  });
  if (attr_err != cudaSuccess) return GS_ERR_CUDA;
  const int kw = ps[0]->g_in;   // one chunk width per launch
  for (int i = 1; i < n; ++i)
    if (ps[i]->g_in != kw) return GS_ERR_UNSUPPORTED;
  if (kw != 128 && kw != 256) return GS_ERR_UNSUPPORTED;
  // Up to 128 tokens a pair tile (256 tokens) would be half empty: each CTA
  // then takes a 128-token tile of its own.
  const bool pair = T > kBM;
  const int64_t tile_m = pair ? kPairM : kBM;
  // Layers with no kept group produce zeros; the others share launches of up
  // to kMaxLayers, largest work per tile (kept groups per window) first, so
  // the last tiles the pairs pick up are the short ones.
  std::vector<int> order;
  for (int i = 0; i < n; ++i) {
    const gs_packed* p = ps[i];
    if (p->kept == 0) {
      if (cudaMemsetAsync(ys[i], 0, (size_t)T * (size_t)p->out * 2, s) != cudaSuccess) return GS_ERR_CUDA;
      continue;
    }
    if (!p->wmaps_valid) return GS_ERR_CUDA;
    if (p->G > kMaxG) return GS_ERR_UNSUPPORTED;
    order.push_back(i);
  }
  auto tile_work = [&](int i) {
    const gs_packed* p = ps[i];
    return (double)p->kept / (double)((p->out + kFW - 1) / kFW);
  };
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return tile_work(a) > tile_work(b); });
  int* err = device_error_flag();
  if (!err) return GS_ERR_CUDA;
  const int64_t max_pairs = sm_count() / 2;
  for (size_t b0 = 0; b0 < order.size(); b0 += kMaxLayers) {
    const int nb = (int)std::min<size_t>(kMaxLayers, order.size() - b0);
    PrefillParams P;
    std::memset(&P, 0, sizeof(P));
    int64_t tiles = 0;
    for (int k = 0; k < nb; ++k) {
      const int i = order[b0 + k];
      const gs_packed* p = ps[i];
      PrefillLayer& L = P.L[k];
      if (!encode_tmap_slabs_bf16(&L.xmap, xs[i], (uint64_t)p->in, (uint64_t)T, kBM, kSlabs)) return GS_ERR_CUDA;
      for (int h = 0; h < kNMaps; ++h) std::memcpy(&L.wmap[h], pair ? p->wmaps[h] : p->wmaps_full[h], sizeof(CUtensorMap));
      L.win_off16 = p->win_off16;
      L.kmask16 = p->kmask16;
      L.y = static_cast<uint16_t*>(ys[i]);
      L.out = (int32_t)p->out;
      L.G = p->G;
      L.nw16 = p->nw16;
      L.n_m = (int32_t)((T + tile_m - 1) / tile_m);
      L.n_w = (int32_t)((p->out + kFW - 1) / kFW);
      L.tile_begin = (int32_t)tiles;
      tiles += (int64_t)L.n_m * L.n_w;
    }
    if (tiles > INT32_MAX) return GS_ERR_UNSUPPORTED;
    P.n_layers = nb;
    P.T = (int32_t)T;
    P.n_tiles = (int32_t)tiles;
    P.err = err;
    P.inject_ns = b0 == 0 ? take_injected_wait(GS_ALGO_PREFILL) : 0;
    const int owners = (int)std::min<int64_t>(tiles, pair ? max_pairs : (int64_t)sm_count());
    if (tiles <= kTileListMax) {
      // a tile's time follows its chunk count (measured flat in density)
      std::vector<int32_t> cost((size_t)tiles);
      for (int k = 0; k < nb; ++k)
        for (int64_t t = 0; t < (int64_t)P.L[k].n_m * P.L[k].n_w; ++t) cost[(size_t)(P.L[k].tile_begin + t)] = P.L[k].G;
      plan_tiles(cost, owners, P.tl);
    }
    cudaError_t e;
    if (pair) {
      const int grid = 2 * owners;   // CTA pairs: clusters of two
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3((unsigned)grid);
      cfg.blockDim = dim3(kThreads);
      cfg.dynamicSmemBytes = kSmemBytes;
      cfg.stream = s;
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = 2;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      e = kw == 256 ? cudaLaunchKernelEx(&cfg, k_prefill<true, 256>, P) : cudaLaunchKernelEx(&cfg, k_prefill<true, 128>, P);
    } else {
      const int grid = owners;
      if (kw == 256) k_prefill<false, 256><<<grid, kThreads, kSmemBytesSingle, s>>>(P);
      else k_prefill<false, 128><<<grid, kThreads, kSmemBytesSingle, s>>>(P);
      e = cudaGetLastError();
    }
    note_launch();
    if (e != cudaSuccess) return GS_ERR_CUDA;
  }
  return GS_OK;
}

gs_status launch_prefill(const void* x, const gs_packed* p, int64_t T, void* y, cudaStream_t s) {
  return launch_prefill_batched(&x, &p, 1, T, &y, s);
}

}  // namespace gs
