// Prefill-regime group-sparse linear with zero-filled windows (1 x 256 and
// 1 x 128 groups, Eq. 1), for layers whose kept fraction is high enough that
// multiplying the pruned rows by zero costs less than gathering the kept ones.
//
// A unit of work is 256 tokens x a window of 256 output rows, owned by a
// cluster of two CTAs: CTA r holds tokens 128 r .. 128 r + 127 and window rows
// 128 r .. 128 r + 127.  For every chunk with a kept row in the window and every
// 64-wide k slab of it, the producer warps place the window's rows in shared
// memory at their row positions (a 16-byte cp.async per piece from the packed
// tiles for a kept row; zeros for a pruned row), next to one TMA box of the
// tokens' x slab, and the leader issues M = 256, N = 256 cta_group::2 MMAs that
// accumulate the whole unit in TMEM.  Nothing is gathered or scattered: the
// accumulator is read once per unit.  Packed weights are read from memory once
// per unit (pruned groups move no bytes); the tensor work is that of the dense
// window, i.e. 1 / density times the kept work.
//
// Roles (one CTA per SM, units persistent over the pairs): warps 0..3
// producers (warp-cooperative 16-byte cp.async of the window's rows, zero-filled
// for pruned rows), warp 4 TMEM allocator + single-thread MMA issuer (leader),
// warps 5..8 epilogue, warp 9 and warps 11.. forwarders (stage pairs taken in
// turn), warp 10 x producer (TMA).  W slots
// and x slots are two rings: the W ring (ten 16 KB slots) runs deeper than
// the x ring (four), because a W slot's round trip (copies landing,
// fences, arrival at the leader) is about three times a TMA's.  Two
// consecutive stages share one readiness barrier (both forwarders, both CTAs'
// x bytes) and one completion barrier: the single MMA-issuing thread spends
// most of a stage on its own instructions (about 40 ns per MMA, 50 per commit
// and 60 per wait), so one wait and one commit per stage pair (eight MMAs)
// instead of two of each per stage took the 13824 x 5120 layer from 1120 to
// ~1220 dense-equivalent TFLOP/s (1 x 256) and 1 x 128 groups from 0.283 to
// 0.232 ms; a second forwarder (the fences of one batch take about a
// microsecond, which one forwarder could no longer hide) then took it to 1440.  Every item therefore has an even number of stages (square groups
// use 128-column items, two slabs with their own tile lookups).  Producers never wait for their own copies: each thread's copies
// of a stage signal a local barrier (cp.async.mbarrier.arrive), and the
// forwarder, once all have landed, fences them to the async proxy and arrives
// on the leader's full barrier.  Every wait is bounded.
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

constexpr int kDM = 128;                          // tokens per CTA (TMEM lanes); a pair covers 256
constexpr int kDW = 256;                          // output rows per window (N of each MMA)
constexpr int kDHalf = kDW / 2;                   // window rows each CTA holds
constexpr int kDSlabK = 64;                       // k per stage (one 128-byte swizzle row)
constexpr int kDXBytes = kDM * kDSlabK * 2;       // 16 KB of x per stage
constexpr int kDWBytes = kDHalf * kDSlabK * 2;    // 16 KB of W rows per stage
// Two rings: W slots (the long round trip: copies landing, forwarder fences,
// arrival at the leader) run deeper than x slots (TMA); with single stages 9 / 3
// measured ahead of 8 / 4, 7 / 5 and 10 / 2; with stage pairs both counts are
// even and the shared memory (224 KB) is used up.
constexpr int kDWStages = 10;                    // 160 KB
constexpr int kDXStages = 4;                     // 64 KB
constexpr int kDSuper = kDWStages / 2;          // pairs of consecutive stages share their barriers
constexpr int kDXRing = kDXStages * kDXBytes;     // 64 KB at offset 0
constexpr int kDWRing = kDWStages * kDWBytes;     // 128 KB after it
constexpr int kDProdWarps = 4;                   // warps that copy W rows
constexpr int kDMmaWarp = kDProdWarps;
constexpr int kDEpiWarp0 = kDProdWarps + 1;
constexpr int kDEpiWarps = 4;
constexpr int kDFwdWarp = kDEpiWarp0 + kDEpiWarps;
constexpr int kDXWarp = kDFwdWarp + 1;            // x TMA producer
constexpr int kDNumFwd = 2;                       // forwarders: warp kDFwdWarp, then kDXWarp + 1, ...
constexpr int kDThreads = (kDXWarp + kDNumFwd) * 32;
constexpr int kDAccBufs = 2;
constexpr uint32_t kDTmemCols = kDAccBufs * kDW;  // 512
constexpr int kDMaxLayers = 8;
constexpr uint64_t kDWaitLimitNs = 2000000000ull;
constexpr uint64_t kDDrainLimitNs = 200000000ull;
constexpr int kDIbufBytes = 1024;                // per-warp chunk lists of d_items
constexpr int kDSmem = kDXRing + kDWRing + kDIbufBytes + 1024;
static_assert(kDHalf % (kDProdWarps * 32) == 0, "producer warps split the CTA's window rows evenly");
static_assert(kDSmem <= 227 * 1024, "shared memory budget");
static_assert(kDWBytes % 1024 == 0 && kDXBytes % 1024 == 0, "slots keep 1024-byte alignment");

struct DLayer {
  CUtensorMap xmap;          // x as (64, T, in/64) slabs, box 64 x 128 x 1
  const uint16_t* tiles;     // 1 x KW: [kept][KW]; square g x g: [kept][g][g]
  const int32_t* win_off16;  // 1 x KW: [G][nw16 + 1]
  const uint16_t* kmask16;   // 1 x KW: [G][nw16]
  const int32_t* gtidx;      // square: [out / g][in / g] packed tile of each group, -1 if pruned
  uint16_t* y;
  int32_t out, G, nw16, n_m, tile_begin;   // G: chunks of KW columns (square: 64-column slabs)
  int32_t Gin;               // square: in / g
};
struct DParams {
  DLayer L[kDMaxLayers];
  int32_t n_layers, T, n_tiles;
  int* err;
  uint64_t inject_ns;   // test hook: CTA pair 0 first waits this long on a word nothing sets (0 = off)
  TileList tl;          // which pair takes which units
};

__device__ __forceinline__ int d_layer_of(const DParams& P, int t) {
  int l = 0;
  while (l + 1 < P.n_layers && P.L[l + 1].tile_begin <= t) ++l;
  return l;
}

// 16-byte copy global -> shared; src_bytes < 16 fills the rest with zeros (0: reads nothing)
__device__ __forceinline__ void cp_async16_zfill(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
// arrive on a local mbarrier once all of this thread's earlier cp.async copies have landed
// (without raising its expected count: the barrier counts the arriving threads)
__device__ __forceinline__ void cp_async_arrive_noinc(uint64_t* bar) {
  asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }
__device__ __forceinline__ void fence_acq_rel_cluster() { asm volatile("fence.acq_rel.cluster;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy_async_cta() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Chunks c0 .. c0 + 31 with at least one kept row in window w, in order, into
// buf (square groups: every 128-column item)
template <int SQ>
__device__ __forceinline__ int d_items(const DLayer& L, int w, int c0, int lane, int16_t* buf) {
  const int c = c0 + lane;
  __syncwarp();   // every lane is done reading the previous batch
  bool ne = false;
  if (c < L.G) {
    if constexpr (SQ > 0) {
      ne = true;
    } else {
      const int32_t* wo = L.win_off16 + (int64_t)c * (L.nw16 + 1);
      const int lo = w * (kDW / kWin16), hi = min(lo + kDW / kWin16, L.nw16);
      ne = wo[hi] > wo[lo];
    }
  }
  const uint32_t ballot = __ballot_sync(0xffffffffu, ne);
  if (ne) buf[__popc(ballot & ((1u << lane) - 1u))] = (int16_t)c;
  __syncwarp();
  return __popc(ballot);
}

__device__ __forceinline__ uint32_t d_pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// KW: chunk width (1 x KW groups; 128 for square groups: items of two slabs);
// SQ: 0, or g for square g x g groups
template <int KW, int SQ>
__global__ void __launch_bounds__(kDThreads, 1) k_prefill_dense(const __grid_constant__ DParams P) {
  constexpr int kSlabs = KW / kDSlabK;   // stages per chunk
  static_assert(kSlabs % 2 == 0 && kDWStages % 2 == 0 && kDXStages % 2 == 0, "stages go in pairs");
  extern __shared__ uint8_t d_smem_raw[];
  // Stage k uses W slot k % kDWStages and x slot k % kDXStages; one barrier of
  // each kind per W slot, so the MMA thread waits once and commits once a stage.
  __shared__ __align__(8) uint64_t full_bar[kDSuper];       // leader: both forwarders + both CTAs' x bytes, two stages
  __shared__ __align__(8) uint64_t done_bar[kDSuper];       // the two stages' MMAs completed (both CTAs)
  __shared__ __align__(8) uint64_t wfull_bar[kDWStages];    // local: this CTA's producer threads' copies
  __shared__ __align__(8) uint64_t afull_bar[kDAccBufs];
  __shared__ __align__(8) uint64_t aempty_bar[kDAccBufs];
  __shared__ __align__(8) uint64_t drain_bar;
  __shared__ uint32_t tmem_base_s;
  __shared__ int abort_s;
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(d_smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();   // 0: leader (issues the pair's MMAs)
  // chunk lists of d_items (producers, MMA issuer, x producer, forwarders)
  const int ib_slot = warp <= kDMmaWarp ? warp : warp == kDFwdWarp ? kDMmaWarp + 1 : warp >= kDXWarp ? warp - kDXWarp + kDMmaWarp + 2 : 0;
  int16_t* ibuf = reinterpret_cast<int16_t*>(smem + kDXRing + kDWRing) + ib_slot * 32;
  static_assert((kDMmaWarp + 2 + kDNumFwd) * 32 * 2 <= kDIbufBytes, "chunk lists fit");

  if (threadIdx.x == 0) {
    for (int s = 0; s < kDSuper; ++s) {
      mbar_init(&full_bar[s], 2 * (2 + 1));   // per stage: both CTAs' forwarders + the leader's expect-tx
      mbar_init(&done_bar[s], 1);
    }
    for (int s = 0; s < kDWStages; ++s) mbar_init(&wfull_bar[s], kDProdWarps * 32);
    for (int b = 0; b < kDAccBufs; ++b) {
      mbar_init(&afull_bar[b], 1);
      mbar_init(&aempty_bar[b], 2 * kDEpiWarps);
    }
    mbar_init(&drain_bar, 1);
    abort_s = 0;
    fence_mbar_init();
    for (int l = 0; l < P.n_layers; ++l) prefetch_tmap(&P.L[l].xmap);
  }
  if (warp == kDMmaWarp) {
    tmem_alloc_pair(&tmem_base_s, kDTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync_all();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  volatile int* abort_flag = &abort_s;
  const int n_tiles = P.n_tiles;
  const int pair = (int)(blockIdx.x >> 1), n_pairs = (int)(gridDim.x >> 1);

  if (P.inject_ns != 0 && pair == 0) {
    // test hook: before any copy or MMA is issued, a bounded wait on a word
    // that nothing sets runs out in each CTA of pair 0; the pair then records
    // the timeout and skips its units (every role, both CTAs)
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
  } else if (warp < kDProdWarps) {
    // ------------------------------------------------------------ producers
    // Warp v copies window rows v * kRows .. + kRows - 1 of this CTA's half,
    // warp-cooperatively: copy i moves rows v * kRows + 4 i .. + 3, eight
    // lanes per 128-byte row, so each instruction reads four whole lines.
    // Lane l looks up the packed positions of rows v * kRows + 32 q + l.
    constexpr int kRows = kDHalf / kDProdWarps;   // rows per producer warp
    constexpr int kOwn = kRows / 32;              // rows whose metadata a lane loads
    constexpr int kCopies = kRows / 4;            // 16-byte copies per lane per stage
    uint32_t stage = 0, phase = 0;
    bool ok = true;
    for (int ku = 0, u; ok && (u = owner_tile(P.tl, n_tiles, pair, n_pairs, ku)) >= 0; ++ku) {
      const DLayer& L = P.L[d_layer_of(P, u)];
      const int w = (u - L.tile_begin) / L.n_m;
      const int j = lane & 7;   // 16-byte piece of a row this lane copies
      // 1 x KW: metadata of this lane's rows in chunk c, the window's kept mask
      // and first packed row (two independent loads, issued one item ahead of use)
      auto load_meta = [&](int c, uint32_t (&km)[kOwn], int (&wo)[kOwn]) {
#pragma unroll
        for (int q = 0; q < kOwn; ++q) {
          const int h = (int)rank * kDHalf + warp * kRows + 32 * q + lane;   // row within the window
          const int b16 = min(w * (kDW / kWin16) + (h >> 4), L.nw16 - 1);
          km[q] = L.kmask16[(int64_t)c * L.nw16 + b16];
          wo[q] = L.win_off16[(int64_t)c * (L.nw16 + 1) + b16];
        }
      };
      // square: packed tile of each piece this lane copies in each slab of item c
      // (its row's block row, its columns' block column), loaded one item ahead
      constexpr int kTS = SQ > 0 ? kSlabs : 1;   // slabs with their own tile lookups
      // a warp's 32 rows lie in one block row (g >= 32) or two (g = 16): one
      // lookup per block row and slab; copy i uses block row kU * i / kCopies
      constexpr int kU = SQ == 16 ? 2 : 1;
      auto load_tiles = [&](int c, int (&tv)[kTS][kU]) {
#pragma unroll
        for (int sl = 0; sl < kTS; ++sl)
#pragma unroll
          for (int q = 0; q < kU; ++q) {
            const int row = w * kDW + (int)rank * kDHalf + warp * kRows + 16 * q;   // first row of the block row part
            const int k = c * KW + sl * kDSlabK + 8 * j;
            tv[sl][q] = row < L.out ? L.gtidx[(int64_t)(row / (SQ > 0 ? SQ : 1)) * L.Gin + k / (SQ > 0 ? SQ : 1)] : -1;
          }
      };
      for (int c0 = 0; c0 < L.G && ok; c0 += 32) {
        const int n_it = d_items<SQ>(L, w, c0, lane, ibuf);
        uint32_t km_n[kOwn];
        int wo_n[kOwn];
        int tv_n[kTS][kU];
        if (n_it > 0) {
          if constexpr (SQ > 0) load_tiles(ibuf[0], tv_n);
          else load_meta(ibuf[0], km_n, wo_n);
        }
        for (int it = 0; it < n_it && ok; ++it) {
          const int c = ibuf[it];
          // element offset of each piece this lane copies (1 x KW: slab 0 of the
          // item, the others follow at 64-element steps; square: per slab), -1: zeros
          int64_t soff[kTS][kCopies];
          if constexpr (SQ > 0) {
#pragma unroll
            for (int sl = 0; sl < kTS; ++sl)
#pragma unroll
              for (int i = 0; i < kCopies; ++i) {
                const int row = w * kDW + (int)rank * kDHalf + warp * kRows + 4 * i + (lane >> 3);
                const int k = c * KW + sl * kDSlabK + 8 * j;
                const int tq = tv_n[sl][kU * i / kCopies];
                soff[sl][i] = tq >= 0 ? ((int64_t)tq * SQ + row % SQ) * SQ + k % SQ : -1;
              }
            if (it + 1 < n_it) load_tiles(ibuf[it + 1], tv_n);
          } else {
            // packed positions in chunk c of the rows this lane looks up (-1: pruned / beyond out)
            int prow[kOwn];
#pragma unroll
            for (int q = 0; q < kOwn; ++q) {
              const int h = (int)rank * kDHalf + warp * kRows + 32 * q + lane;
              const int b16 = w * (kDW / kWin16) + (h >> 4), bit = h & 15;
              const bool kept = b16 < L.nw16 && ((km_n[q] >> bit) & 1u);
              prow[q] = kept ? wo_n[q] + __popc(km_n[q] & ((1u << bit) - 1u)) : -1;
            }
            if (it + 1 < n_it) load_meta(ibuf[it + 1], km_n, wo_n);
            // the rows this lane copies: warp * kRows + 4 i + (lane >> 3)
#pragma unroll
            for (int i = 0; i < kCopies; ++i) {
              const int r = 4 * i + (lane >> 3);   // row within the warp's block: owner lane r % 32, slot r / 32
              const int pr = __shfl_sync(0xffffffffu, prow[r >> 5], r & 31);
              soff[0][i] = pr >= 0 ? (int64_t)pr * KW + 8 * j : -1;
            }
          }
#pragma unroll
          for (int sl = 0; sl < kSlabs; ++sl) {
            if (!ok) break;
            bool got = true;
            if (lane == 0)
              got = mbar_wait_bounded(&done_bar[stage / 2], phase ^ 1u, abort_flag, P.err, kDWaitLimitNs, kDevErrTimeout);
            if (!__shfl_sync(0xffffffffu, got ? 1 : 0, 0)) {
              ok = false;
              break;
            }
            const uint32_t wb = smem_u32(smem + kDXRing + stage * kDWBytes);
#pragma unroll
            for (int i = 0; i < kCopies; ++i) {
              const int rr = warp * kRows + 4 * i + (lane >> 3);
              const uint32_t dst = wb + (uint32_t)rr * 128u + (uint32_t)((j ^ (rr & 7)) << 4);   // 128-byte swizzle
              const int64_t so = soff[SQ > 0 ? sl : 0][i];
              const bool kept = so >= 0;
              // a pruned row reads nothing (source size 0) and is filled with zeros
              const uint16_t* src = kept ? L.tiles + so + (SQ > 0 ? 0 : sl * kDSlabK) : L.tiles;
              cp_async16_zfill(dst, src, kept ? 16u : 0u);
            }
            cp_async_arrive_noinc(&wfull_bar[stage]);   // fires once this thread's copies have landed
            if (++stage == (uint32_t)kDWStages) {
              stage = 0;
              phase ^= 1u;
            }
          }
        }
      }
    }
    cp_async_wait_all();
    __syncwarp();
  } else if (warp == kDXWarp) {
    // ------------------------------------------------------------ x producer
    // Stage k's x box goes to x slot k % kDXStages once stage k - kDXStages is
    // done, and completes on the leader's full barrier of W slot k % kDWStages.
    uint32_t k = 0;
    uint32_t armed = 0u, armed_par = 0u;
    bool ok = true;
    for (int ku = 0, u; ok && (u = owner_tile(P.tl, n_tiles, pair, n_pairs, ku)) >= 0; ++ku) {
      const DLayer& L = P.L[d_layer_of(P, u)];
      const int lt = u - L.tile_begin;
      const int m = lt % L.n_m, w = lt / L.n_m;
      const int tok0 = m * 2 * kDM + (int)rank * kDM;
      for (int c0 = 0; c0 < L.G && ok; c0 += 32) {
        const int n_it = d_items<SQ>(L, w, c0, lane, ibuf);
        if (lane == 0) {
          for (int it = 0; it < n_it && ok; ++it) {
            const int c = ibuf[it];
            for (int sl = 0; sl < kSlabs && ok; ++sl, ++k) {
              if (k >= (uint32_t)kDXStages) {
                const uint32_t pp = (k - kDXStages) / 2;   // the stage pair whose x slot this one reuses
                if (!mbar_wait_bounded(&done_bar[pp % kDSuper], (pp / kDSuper) & 1u, abort_flag, P.err,
                                       kDWaitLimitNs, kDevErrTimeout)) {
                  ok = false;
                  break;
                }
              }
              const uint32_t fs = (k / 2) % kDSuper;
              if (rank == 0) mbar_arrive_expect_tx(&full_bar[fs], 2u * kDXBytes);
              tma_load_3d_pair(smem + (k % kDXStages) * kDXBytes, &L.xmap, mapa_shared(smem_u32(&full_bar[fs]), 0),
                               0, tok0, c * kSlabs + sl);
              armed |= 1u << fs;
              armed_par = (armed_par & ~(1u << fs)) | (((k / 2 / kDSuper) & 1u) << fs);
            }
          }
        }
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      }
    }
    if (lane == 0 && !ok && rank == 0) {
      // let the x copies in flight land before the CTA winds down
      for (int s = 0; s < kDSuper; ++s) {
        if (!((armed >> s) & 1u)) continue;
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait_acq_cluster(&full_bar[s], (armed_par >> s) & 1u))
          if (globaltimer_ns() - t0 > kDDrainLimitNs) break;
      }
    }
    __syncwarp();
  } else if (warp == kDFwdWarp || warp > kDXWarp) {
    // ------------------------------------------------------------ forwarders
    // Once all of this CTA's producer threads' copies of a stage pair have
    // landed, make them visible to the tensor cores (async proxy) and tell the
    // leader.  The forwarders take the stage pairs in turn, so that their
    // fences (about a microsecond per batch) overlap.
    const uint32_t f = warp == kDFwdWarp ? 0u : (uint32_t)(warp - kDXWarp);   // takes pairs p with p % kDNumFwd == f
    uint32_t K = 0;   // stages before the current batch
    bool ok = true;
    for (int ku = 0, u; ok && (u = owner_tile(P.tl, n_tiles, pair, n_pairs, ku)) >= 0; ++ku) {
      const DLayer& L = P.L[d_layer_of(P, u)];
      const int w = (u - L.tile_begin) / L.n_m;
      for (int c0 = 0; c0 < L.G && ok; c0 += 32) {
        const int n_pr = d_items<SQ>(L, w, c0, lane, ibuf) * kSlabs / 2;   // stage pairs of the batch
        if (lane == 0) {
          int cnt = 1;
          for (int q = (int)((f + kDNumFwd - (K / 2) % kDNumFwd) % kDNumFwd); q < n_pr && ok; q += kDNumFwd * cnt) {
            const uint32_t p0 = K / 2 + (uint32_t)q;   // global pair index
            const uint32_t s0 = (2 * p0) % kDWStages, ph0 = ((2 * p0) / kDWStages) & 1u;
            if (!mbar_wait_bounded(&wfull_bar[s0], ph0, abort_flag, P.err, kDWaitLimitNs, kDevErrTimeout) ||
                !mbar_wait_bounded(&wfull_bar[s0 + 1], ph0, abort_flag, P.err, kDWaitLimitNs, kDevErrTimeout)) {
              ok = false;
              break;
            }
            // take this forwarder's following pairs that have landed too, so that
            // one release fence covers them all (a release per stage is slow)
            cnt = 1;
            while (q + kDNumFwd * cnt < n_pr && cnt * kDNumFwd < kDSuper) {
              const uint32_t p2 = p0 + kDNumFwd * (uint32_t)cnt;
              const uint32_t s2 = (2 * p2) % kDWStages, ph2 = ((2 * p2) / kDWStages) & 1u;
              if (!mbar_try_wait(&wfull_bar[s2], ph2) || !mbar_try_wait(&wfull_bar[s2 + 1], ph2)) break;
              ++cnt;
            }
            fence_proxy_async_cta();
            fence_acq_rel_cluster();   // with the relaxed arrives below: a release of the copies to the leader
            for (int i = 0; i < cnt; ++i) {
              const uint32_t fs = (p0 + kDNumFwd * (uint32_t)i) % kDSuper;
              const uint32_t fb = mapa_shared(smem_u32(&full_bar[fs]), 0);
              mbar_arrive_cluster_relaxed(fb);   // one arrival per stage of the pair
              mbar_arrive_cluster_relaxed(fb);
            }
          }
        }
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
        K += (uint32_t)(2 * n_pr);
      }
    }
  } else if (warp == kDMmaWarp && rank == 0) {
    // ------------------------------------------------------------ MMA issuer (leader)
    uint32_t ws = 0, wph = 0, xs = 0;   // W slot (and its barriers' phase), x slot
    int buf = 0;
    uint32_t ae_ph = 0u;
    bool ok = true;
    constexpr uint32_t idesc = idesc_bf16_f32(2 * kDM, kDW);
    for (int ku = 0, u; ok && (u = owner_tile(P.tl, n_tiles, pair, n_pairs, ku)) >= 0; ++ku) {
      const DLayer& L = P.L[d_layer_of(P, u)];
      const int w = (u - L.tile_begin) / L.n_m;
      if (lane == 0) {
        ok = mbar_wait_bounded_cluster(&aempty_bar[buf], ((ae_ph >> buf) & 1u) ^ 1u, abort_flag, P.err, kDWaitLimitNs,
                                       kDevErrTimeout);
        ae_ph ^= 1u << buf;
        tc_fence_after();
      }
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      const uint32_t d = tmem + (uint32_t)(buf * kDW);
      bool first = true;
      for (int c0 = 0; c0 < L.G && ok; c0 += 32) {
        const int n_it = d_items<SQ>(L, w, c0, lane, ibuf);
        if (lane == 0) {
          // stages two at a time (every item has an even number of them)
          for (int it = 0; it < n_it * kSlabs && ok; it += 2) {
            if (!mbar_wait_bounded_cluster(&full_bar[ws / 2], wph, abort_flag, P.err, kDWaitLimitNs, kDevErrTimeout)) {
              ok = false;
              break;
            }
            tc_fence_after();
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const uint64_t ad = sdesc_sw128(smem_u32(smem + (xs + h) * kDXBytes));
              const uint64_t bd = sdesc_sw128(smem_u32(smem + kDXRing + (ws + h) * kDWBytes));
#pragma unroll
              for (int kk = 0; kk < kDSlabK / 16; ++kk)
                mma_bf16_ss_pair(d, ad + (uint64_t)(2 * kk), bd + (uint64_t)(2 * kk), idesc,
                                 (first && h == 0 && kk == 0) ? 0u : 1u);
            }
            first = false;
            mma_commit_pair_mc(&done_bar[ws / 2], 0x3);
            ws += 2;
            if (ws == (uint32_t)kDWStages) {
              ws = 0;
              wph ^= 1u;
            }
            xs += 2;
            if (xs == (uint32_t)kDXStages) xs = 0;
          }
        }
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
        first = __shfl_sync(0xffffffffu, first ? 1 : 0, 0) != 0;
      }
      if (!ok) break;
      if (lane == 0) mma_commit_pair_mc(&afull_bar[buf], 0x3);
      buf ^= 1;
    }
    if (lane == 0) {
      mma_commit_pair(&drain_bar);
      mbar_wait_bounded(&drain_bar, 0u, nullptr, P.err, kDWaitLimitNs, kDevErrTimeout);
    }
    __syncwarp();
  } else if (warp >= kDEpiWarp0) {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;   // TMEM lane quarter this warp may access
    int buf = 0;
    uint32_t af_ph = 0u;
    bool ok = true;
    for (int ku = 0, u; ok && (u = owner_tile(P.tl, n_tiles, pair, n_pairs, ku)) >= 0; ++ku) {
      const DLayer& L = P.L[d_layer_of(P, u)];
      const int lt = u - L.tile_begin;
      const int m = lt % L.n_m, w = lt / L.n_m;
      // a window with no kept row in any chunk has no MMA: its rows are zero
      bool any = SQ > 0;   // square groups: every slab has MMAs
      if constexpr (SQ == 0) {
        const int lo = w * (kDW / kWin16), hi = min(lo + kDW / kWin16, L.nw16);
        for (int c = lane; c < L.G && !any; c += 32) {
          const int32_t* wo = L.win_off16 + (int64_t)c * (L.nw16 + 1);
          any = wo[hi] > wo[lo];
        }
        any = __any_sync(0xffffffffu, any);
      }
      const bool got =
          mbar_wait_bounded(&afull_bar[buf], (af_ph >> buf) & 1u, abort_flag, P.err, kDWaitLimitNs, kDevErrTimeout);
      if (!__all_sync(0xffffffffu, got)) {   // the TMEM loads below need the whole warp
        ok = false;
        break;
      }
      af_ph ^= 1u << buf;
      tc_fence_after();
      const int tok = m * 2 * kDM + (int)rank * kDM + 32 * q + lane;
      uint16_t* yrow = L.y + (int64_t)tok * L.out;
      const bool vec_ok = (L.out & 7) == 0;
#pragma unroll 1
      for (int j = 0; j < kDW / 32; ++j) {
        uint32_t v[32];
        tmem_ld_x32(tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * kDW + 32 * j), v);
        tmem_wait_ld();
        reg_fence(v);
        const int r0 = w * kDW + 32 * j;
        if (tok < P.T) {
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const int rb = r0 + 8 * k;
            const float* f = reinterpret_cast<const float*>(v + 8 * k);
            if (vec_ok && rb + 8 <= L.out) {
              *reinterpret_cast<uint4*>(yrow + rb) =
                  any ? make_uint4(d_pack_bf16x2(f[0], f[1]), d_pack_bf16x2(f[2], f[3]), d_pack_bf16x2(f[4], f[5]),
                                   d_pack_bf16x2(f[6], f[7]))
                      : make_uint4(0u, 0u, 0u, 0u);
            } else {
#pragma unroll
              for (int e = 0; e < 8; ++e)
                if (rb + e < L.out) yrow[rb + e] = any ? __bfloat16_as_ushort(__float2bfloat16_rn(f[e])) : 0;
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster_relaxed(mapa_shared(smem_u32(&aempty_bar[buf]), 0));
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
  cluster_sync_all();
  if (warp == kDMmaWarp) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, kDTmemCols);
  }
  cluster_sync_all();
}

int d_sm_count() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 148;
  }
  return n;
}

template <int KW, int SQ>
cudaError_t d_set_attr() {
  static std::once_flag once;
  static cudaError_t err = cudaSuccess;
  std::call_once(once, []() {
    err = cudaFuncSetAttribute(k_prefill_dense<KW, SQ>, cudaFuncAttributeMaxDynamicSharedMemorySize, kDSmem);
  });
  return err;
}

template <int KW, int SQ>
cudaError_t d_launch(const cudaLaunchConfig_t& cfg, const DParams& P) {
  const cudaError_t e = d_set_attr<KW, SQ>();
  if (e != cudaSuccess) return e;
  return cudaLaunchKernelEx(&cfg, k_prefill_dense<KW, SQ>, P);
}

}  // namespace

// Which 1 x KW layers take this kernel rather than the gathering one, by the
// layer's own group shape and T (so that a batched call gives each layer what
// gs_linear gives it, bit for bit).  Measured on GB300 at d = 0.5 with the
// balanced tile lists, one batched call per block (7 projections):
//  - 1 x 256 from 129 tokens: LLaMA-2-13B block 0.142 / 0.144 / 0.236 / 0.330
//    ms at T = 160 / 256 / 512 / 640 against 0.172 / 0.173 / 0.294 / 0.426 with
//    the gathering kernel for the 5120-row layers (7B block 0.101-0.220 against
//    0.117-0.299; Qwen2.5-7B 0.180-0.249 against 0.217-0.304 from T = 384, 4 %
//    behind at 160 and 256).  Alone, a 5120 x 5120 layer at T = 512 still runs
//    faster gathering (0.040 vs 0.048 ms: 40 units for 76 CTA pairs), but layers
//    are mostly called a block at a time;
//  - 1 x 128 in the whole prefill regime: over the five 7B / 13B projection
//    shapes at T = 64 and 128 it takes 0.91-0.96x the gathering kernel's time in
//    nine of the ten cases (13824 x 5120 at T = 128: 1.02x), while 1 x 256
//    layers up to 128 tokens stay on the gathering kernel (1.15-1.24x).
// Both kernels' times hardly depend on the density.
bool prefill_prefers_dense(const gs_packed* p, int64_t T) {
  if (p->kept == 0 || p->g_out != 1) return false;
  if (p->g_in == 128) return true;
  return p->g_in == 256 && T > 128;
}

gs_status launch_prefill_dense(const void* const* xs, const gs_packed* const* ps, int n, int64_t T, void* const* ys,
                               cudaStream_t s, const int* idx) {
  if (T <= 0 || n <= 0) return GS_OK;
  std::vector<int> order(n);
  for (int i = 0; i < n; ++i) order[i] = idx ? idx[i] : i;
  const int kw = ps[order[0]]->g_in, go = ps[order[0]]->g_out;
  for (int i : order)
    if (ps[i]->g_in != kw || ps[i]->g_out != go || ps[i]->kept == 0) return GS_ERR_UNSUPPORTED;
  const int sq = go > 1 ? go : 0;   // square g x g groups
  if (sq ? (sq != kw || (sq != 16 && sq != 32 && sq != 64)) : (kw != 256 && kw != 128)) return GS_ERR_UNSUPPORTED;
  for (int i : order)
    if (sq && !ps[i]->gtidx) return GS_ERR_UNSUPPORTED;
  int* err = device_error_flag();
  if (!err) return GS_ERR_CUDA;
  // most tensor work per unit (the widest input) first
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return ps[a]->in > ps[b]->in; });
  const int64_t max_pairs = d_sm_count() / 2;
  for (int b0 = 0; b0 < n; b0 += kDMaxLayers) {
    const int nb = std::min(kDMaxLayers, n - b0);
    DParams P;
    std::memset(&P, 0, sizeof(P));
    int64_t tiles = 0;
    for (int k = 0; k < nb; ++k) {
      const int i = order[b0 + k];
      const gs_packed* p = ps[i];
      DLayer& L = P.L[k];
      if (!encode_tmap_slabs_bf16(&L.xmap, xs[i], (uint64_t)p->in, (uint64_t)T, kDM, 1)) return GS_ERR_CUDA;
      L.tiles = p->tiles;
      L.y = static_cast<uint16_t*>(ys[i]);
      L.out = (int32_t)p->out;
      if (sq) {
        if (p->in % 128 != 0) return GS_ERR_UNSUPPORTED;
        L.gtidx = p->gtidx;
        L.Gin = p->G;
        L.G = (int32_t)(p->in / 128);   // 128-column items (two 64-column stages)
      } else {
        L.win_off16 = p->win_off16;
        L.kmask16 = p->kmask16;
        L.G = p->G;
        L.nw16 = p->nw16;
      }
      if (L.G > 32767) return GS_ERR_UNSUPPORTED;   // chunk lists hold 16-bit indices
      L.n_m = (int32_t)((T + 2 * kDM - 1) / (2 * kDM));
      L.tile_begin = (int32_t)tiles;
      tiles += (int64_t)L.n_m * ((p->out + kDW - 1) / kDW);
    }
    if (tiles > INT32_MAX) return GS_ERR_UNSUPPORTED;
    P.n_layers = nb;
    P.T = (int32_t)T;
    P.n_tiles = (int32_t)tiles;
    P.err = err;
    P.inject_ns = b0 == 0 ? take_injected_wait(GS_ALGO_PREFILL_DENSE) : 0;
    const int owners = (int)std::min<int64_t>(tiles, max_pairs);
    if (tiles <= kTileListMax) {
      // a unit's time follows its item count (one launch holds one chunk width)
      std::vector<int32_t> cost((size_t)tiles);
      for (int k = 0; k < nb; ++k) {
        const int64_t nu = (int64_t)P.L[k].n_m * ((ps[order[b0 + k]]->out + kDW - 1) / kDW);
        for (int64_t t = 0; t < nu; ++t) cost[(size_t)(P.L[k].tile_begin + t)] = P.L[k].G;
      }
      plan_tiles(cost, owners, P.tl);
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(2 * owners));
    cfg.blockDim = dim3(kDThreads);
    cfg.dynamicSmemBytes = kDSmem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t e = sq == 16   ? d_launch<128, 16>(cfg, P)
                          : sq == 32 ? d_launch<128, 32>(cfg, P)
                          : sq == 64 ? d_launch<128, 64>(cfg, P)
                          : kw == 256 ? d_launch<256, 0>(cfg, P)
                                      : d_launch<128, 0>(cfg, P);
    note_launch();
    if (e != cudaSuccess) return GS_ERR_CUDA;
  }
  return GS_OK;
}

}  // namespace gs
