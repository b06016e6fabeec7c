// Decode-regime group-sparse linear (few tokens, HBM-bound):
//   y[t, r] = sum over kept groups (r, c) of sum_k x[t, 256c+k] W[r, 256c+k]   (Eq. 1)
//
// Work units.  A unit is (64-row block, range of chunks) of one layer: a
// block's chunks are split into equal ranges of about 224 KB of kept weights
// (a quarter of that when a launch has too few units to spread over the
// CTAs).  Persistent CTA b starts on units b and
// b + grid, then takes units from a shared ticket counter in list order
// (largest layers first), so a CTA that runs ahead takes more units, and the
// pipeline never restarts between units.
//
// Data movement.  Inside a chunk the kept rows of a 64-row block are one
// contiguous slice of the packed tiles, so a producer warp streams each chunk's
// slice with a single bulk copy (cp.async.bulk) into a byte-granular
// shared-memory ring (each chunk takes its x rows + slice, from a 1024-byte
// aligned start, so the ring holds several chunks in flight), and the chunk's
// x rows with one 3-D TMA box: four 64-wide slabs with the 128-byte swizzle,
// which keeps the consumers' x fragment reads free of bank conflicts; only
// kept bytes move.  The
// producer also stages each unit's per-chunk metadata (slice start + the
// 16-bit kept masks of the four 16-row windows).
//
// Compute.  Two consumer warps own each 16-row window w of the block (rows
// 16w..16w+15): one takes the unit's even chunks, the other its odd chunks,
// so two chunks per window are in flight in the MMA pipeline.  A warp builds
// mma.sync A fragments from the slice, placing every kept row at its window
// position (pruned rows stay zero), with the x chunk as the B fragment.  The
// MMA row is the output row, so the fp32 accumulator stays in registers for
// the whole unit: no scatter and no atomics on y.  At the unit's end one warp
// of the pair hands its accumulator to the other through shared memory, which
// adds it (one fp32 add per element) and writes the result; the writing role
// alternates between the two warps from unit to unit.
//
// Reduction.  When a block's chunks are split over several units, the
// writing warp of each window writes its 16-row partial to the handle's
// workspace and bumps the window's arrival counter; the last arriver adds the
// partials in split order (so the result does not depend on arrival order),
// writes y and resets the counter.
//
// K permutation.  At step b (0..7) lane (g, q) holds the eight consecutive
// weights of 16-byte chunk j = 8(b>>1) + 2q + (b&1) of rows g and g+8 (k = 8j
// + 0..7) and the same eight x values of token g.  Elements 0..3 feed MMA 2b,
// elements 4..7 feed MMA 2b+1; the logical-to-physical k map depends only on
// (b, q), so A and B agree and every physical k is used exactly once.  The
// four q lanes of a token read every other chunk of a 128-byte slab row, so
// after the swizzle (chunk ^ row&7) tokens 2p and 2p+1, which share a
// quarter-warp load phase, land on disjoint banks.
#include "gs_common.cuh"
#include "gs_sm100.cuh"

#include <cuda.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>
#include <vector>

namespace gs {
namespace {
using namespace sm100;

constexpr int kDW = 4;                        // 16-row windows per block
constexpr int kCW = 2 * kDW;                  // consumer warps: two per window (even / odd chunks)
constexpr int kRows = kDW * kWin16;           // 64 rows per block
constexpr int kThreadsDec = (kCW + 1) * 32;   // + one producer warp
constexpr int kMaxNT = 2;                     // 8-token MMA tiles per launch
constexpr int kMaxBatch = 32;
constexpr int kSmallBatch = 8;
constexpr int kMaxT = 16;                     // tokens per launch (two 8-token MMA tiles)
constexpr int kRingBytes = 104 * 1024;       // byte ring per CTA (two CTAs per SM)
constexpr int kRingSeq = 16;                  // chunks that may be in flight (barrier ring)
constexpr int kXRow = kTileBytes;             // x chunk row (512 B): one 3-D TMA box of 4 swizzled 64-wide slabs per chunk
constexpr int kMaxCpu = 64;                   // chunks per unit
constexpr int kMetaSlots = 2;
constexpr int kDecSmemBytes = kRingBytes + kMetaSlots * kMaxCpu * 16 + 1024;
constexpr int kPartFloats = kMaxT * kWin16;   // one warp's partial: 16 tokens x 16 rows
constexpr int64_t kUnitBytes = 224 * 1024;    // target kept bytes per unit
// Ring allocation never waits forever: a chunk that does not fit before the
// ring's end starts over at offset 0, which with every earlier chunk released
// asks for (ring end - head) + need bytes; that stays within the ring for any
// head only while two largest chunks (all 64 rows kept, kMaxT x rows) plus the
// 1024-byte alignment fit in it.
static_assert(2 * (kRows * kTileBytes + kMaxT * kXRow) + 1023 <= kRingBytes,
              "decode ring must hold two largest chunks plus alignment");
constexpr uint64_t kDecWaitLimitNs = 2000000000ull;
constexpr uint64_t kDecDrainLimitNs = 200000000ull;

struct DecLayer {
  CUtensorMap xmap;      // x [T][in] as (64, T, in/64) slabs, box 64 x T x 4, 128-byte swizzle
  const uint16_t* x;     // [T][in]
  const uint16_t* tiles; // [kept][chunk width]
  const int4* dmeta;     // [nblk][G]
  uint16_t* y;           // [T][out]
  float* ws;             // [nblk][nsplit][4][kPartFloats]
  int32_t* cnt;          // [nblk][4]
  int32_t out, in, G, nblk, cpu, nsplit;
  int32_t unit_begin;
};

// Launch parameters for up to MB layers.  Launches of at most kSmallBatch
// layers use the small instance: the parameter block (about 256 B per layer)
// is copied with every launch.
template <int MB>
struct DecParams {
  DecLayer L[MB];
  int32_t n_layers;
  int32_t T;
  int32_t n_units;
  int32_t* sched;        // {next unit ticket, finished CTAs}: zero between launches
  int* err;
  uint64_t inject_ns;    // test hook: CTA 0 first waits this long on a word nothing sets (0 = off)
};

// Weight slices are read once per launch: the evict-first L2 policy keeps
// them from displacing what is reused (x, chunk metadata, split workspace).
__device__ __forceinline__ void bulk_copy_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;"
      ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(pol)
      : "memory");
}

// bulk prefetch of [p, p + bytes) into L2 (bytes a multiple of 16)
__device__ __forceinline__ void prefetch_l2_bulk(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

// atomic add with acquire-release ordering at GPU scope; returns the old value
__device__ __forceinline__ int atom_add_acq_rel_gpu(int32_t* p, int v) {
  int old;
  asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint16_t f32_to_bf16_rn(float f) { return __bfloat16_as_ushort(__float2bfloat16_rn(f)); }

// kept mask of window w (0..3) from a metadata entry
__device__ __forceinline__ uint32_t meta_mask(const int4& m, int w) {
  const uint32_t v = (uint32_t)(w < 2 ? m.y : m.z);
  return (w & 1) ? (v >> 16) : (v & 0xFFFFu);
}

struct Unit {
  int l, blk, c0, nC;
};

// unit u of the launch's unit list; lay[l] = {first unit, splits per block,
// chunks per unit, chunks} of layer l, staged in shared memory
__device__ __forceinline__ void unit_at(const int4* lay, int n_layers, int u, Unit& U) {
  int l = 0;
  while (l + 1 < n_layers && lay[l + 1].x <= u) ++l;
  const int4 L = lay[l];
  const int r = u - L.x;
  U.l = l;
  U.blk = r / L.y;
  const int split = r - U.blk * L.y;
  U.c0 = split * L.z;
  U.nC = min(L.w, U.c0 + L.z) - U.c0;
}

// KW = chunk width: 256 (1 x 256 groups) or 128 (1 x 128 groups)
template <int NT, int MB, int KW>
__global__ void __launch_bounds__(kThreadsDec, 2) k_decode(const __grid_constant__ DecParams<MB> P) {
  static_assert(KW == 128 || KW == 256, "chunk width");
  extern __shared__ uint8_t dsmem_raw[];
  __shared__ __align__(8) uint64_t w_full[kRingSeq];
  __shared__ __align__(8) uint64_t w_empty[kRingSeq];
  __shared__ uint32_t w_off[kRingSeq];   // ring offset of each in-flight chunk
  __shared__ uint32_t w_end[kRingSeq];   // its virtual end offset (producer bookkeeping)
  __shared__ __align__(8) uint64_t m_full[kMetaSlots];
  __shared__ __align__(8) uint64_t m_empty[kMetaSlots];
  __shared__ int unit_id[kMetaSlots];   // unit staged in each metadata slot (-1: no more units)
  __shared__ int abort_s;
  __shared__ __align__(8) uint64_t p_full[kDW];    // pair hand-off per window: accumulator written
  __shared__ __align__(8) uint64_t p_empty[kDW];   // ... and consumed
  __shared__ __align__(16) float pair_buf[kDW * 32 * 4 * kMaxNT];
  __shared__ int4 lay[MB];                      // per layer: {first unit, splits per block, chunks per unit, chunks}
  __shared__ const int4* lay_dmeta[MB];         // per layer: chunk metadata
  uint8_t* ring = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dsmem_raw) + 1023) & ~uintptr_t(1023));
  int4* meta = reinterpret_cast<int4*>(ring + kRingBytes);   // [kMetaSlots][kMaxCpu]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int k = 0; k < kRingSeq; ++k) {
      mbar_init(&w_full[k], 1);
      mbar_init(&w_empty[k], kDW);
    }
    for (int k = 0; k < kMetaSlots; ++k) {
      mbar_init(&m_full[k], 1);
      mbar_init(&m_empty[k], kCW);
    }
    for (int k = 0; k < kDW; ++k) {
      mbar_init(&p_full[k], 1);
      mbar_init(&p_empty[k], 1);
    }
    abort_s = 0;
    fence_mbar_init();
  }
  if (threadIdx.x < P.n_layers) {
    const DecLayer& L = P.L[threadIdx.x];
    lay[threadIdx.x] = make_int4(L.unit_begin, L.nsplit, L.cpu, L.G);
    lay_dmeta[threadIdx.x] = L.dmeta;
  }
  if (P.inject_ns != 0 && blockIdx.x == 0 && threadIdx.x == 0) {
    // test hook: a bounded wait on a word that nothing sets (the flag word
    // after the error flag) runs out before this CTA issues anything; the CTA
    // then records the timeout and skips all its units
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
  const bool injected_abort = abort_s != 0;
  // Programmatic dependent launch: the next launch in the stream may become
  // resident as soon as SM slots free up.  Before touching anything the grid
  // before it may write (x may be its y; the ticket counter and split
  // workspace may be shared with it) a thread waits for that grid to complete
  // (griddepcontrol.wait).  The packed tiles and chunk metadata are never
  // written by a decode launch, so the producer streams its first unit's
  // weight slices before it waits, overlapping the previous launch's end.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  volatile int* abort_flag = &abort_s;
  const int T = P.T;

  if (injected_abort) {
    // nothing was issued: fall through to the end of the launch
  } else if (warp == kCW) {
    // ------------------------------------------------------------ producer warp
    uint32_t q = 0;              // chunks issued so far (ring sequence number)
    uint32_t oldest = 0;         // oldest chunk not yet known to be released
    // Ring bookkeeping in 32-bit virtual byte offsets: `head` / `tail` =
    // allocated / released, `hoff` = head's offset inside the ring.  Only
    // differences below the ring size are ever taken, so the counters may wrap.
    uint32_t head = 0, tail = 0, hoff = 0;
    bool ok = true;
    // CTA b starts with units b and b + grid; every later unit comes from the
    // launch's ticket counter (ticket t = unit 2 grid + t).  `t_ahead` holds
    // the unit after next: its ticket is taken two units early, so neither the
    // start of the launch nor the atomic's round trip delays any copies.
    const int n_static = 2 * (int)gridDim.x;
    int u = (int)blockIdx.x;
    int t_ahead = (int)(blockIdx.x + gridDim.x);
    bool have = u < P.n_units;
    Unit U{0, 0, 0, 0};
    if (have) unit_at(lay, P.n_layers, u, U);
    // Chunks of the first unit issued before the dependency wait: their x
    // boxes follow once it returns (lane 0; `dep` = wait done).
    bool dep = false;
    uint32_t n_pend = 0;
    int4 pre[kMaxCpu / 32];      // this lane's metadata entries of the next unit to stage
    auto prefetch = [&](const Unit& V, bool hv) {
#pragma unroll
      for (int j = 0; j < kMaxCpu / 32; ++j) {
        const int i = lane + 32 * j;
        pre[j] = (hv && i < V.nC) ? __ldg(lay_dmeta[V.l] + (int64_t)V.blk * lay[V.l].w + V.c0 + i)
                                  : make_int4(0, 0, 0, 0);
      }
    };
    prefetch(U, have);
    for (int k = 0; ok; ++k) {
      const int ms = k % kMetaSlots;
      if (!mbar_wait_bounded(&m_empty[ms], ((uint32_t)(k / kMetaSlots) & 1u) ^ 1u, abort_flag, P.err,
                             kDecWaitLimitNs, kDevErrTimeout)) {
        ok = false;
        break;
      }
      if (!have) {
        // no more units: tell the consumers
        if (lane == 0) {
          unit_id[ms] = -1;
          __threadfence_block();
          mbar_arrive(&m_full[ms]);
        }
        __syncwarp();
        break;
      }
      int4* mrow = meta + ms * kMaxCpu;
#pragma unroll
      for (int j = 0; j < kMaxCpu / 32; ++j)
        if (lane + 32 * j < U.nC) mrow[lane + 32 * j] = pre[j];
      if (k == 0) {
        // Before the grid-dependency wait the first unit's weight slices are
        // also fetched into L2 (the ring takes only its first few chunks), so a
        // CTA that starts while the previous grid is still finishing puts the
        // idle HBM bandwidth of that grid's last units to use.
        const uint16_t* tl = P.L[U.l].tiles;
#pragma unroll
        for (int j = 0; j < kMaxCpu / 32; ++j) {
          if (lane + 32 * j < U.nC) {
            const int4 mp = pre[j];
            const uint32_t cnt = __popc((uint32_t)mp.y) + __popc((uint32_t)mp.z);
            if (cnt) prefetch_l2_bulk(tl + (int64_t)mp.x * KW, cnt * (uint32_t)(2 * KW));
          }
        }
      }
      if (lane == 0) unit_id[ms] = u;
      __threadfence_block();
      __syncwarp();
      if (lane == 0) mbar_arrive(&m_full[ms]);   // release: the staged entries are visible to consumers
      const int u_next = __shfl_sync(0xffffffffu, t_ahead, 0);
      if (lane == 0 && dep && u_next < P.n_units) t_ahead = n_static + atomicAdd(P.sched, 1);
      const bool have_v = u_next < P.n_units;
      Unit V{0, 0, 0, 0};
      if (have_v) unit_at(lay, P.n_layers, u_next, V);
      prefetch(V, have_v);                       // in flight while this unit's copies are issued
      if (lane == 0) {
        const DecLayer& L = P.L[U.l];
        const uint32_t xbytes = (uint32_t)T * (uint32_t)(2 * KW);
        // first unit only: wait for the previous grid, then issue the pending
        // x boxes and take the ticket of the unit after next
        auto resolve = [&]() {
          asm volatile("griddepcontrol.wait;" ::: "memory");
          for (uint32_t i = 0; i < n_pend; ++i) {
            const int4 mp = mrow[i];
            if ((mp.y | mp.z) != 0)
              tma_load_3d(ring + w_off[i], &L.xmap, &w_full[i], 0, 0, (U.c0 + (int)i) * (KW / 64));
          }
          if (u_next < P.n_units) t_ahead = n_static + atomicAdd(P.sched, 1);
          dep = true;
        };
        int4 m_next = U.nC > 0 ? mrow[0] : make_int4(0, 0, 0, 0);
        for (int i = 0; i < U.nC && ok; ++i, ++q) {
          const int4 m = m_next;
          if (i + 1 < U.nC) m_next = mrow[i + 1];
          const uint32_t cnt = __popc((uint32_t)m.y) + __popc((uint32_t)m.z);
          const uint32_t bytes = cnt * (uint32_t)(2 * KW);
          const uint32_t need = cnt ? bytes + xbytes : 0u;
          // allocate `need` contiguous bytes from a 1024-byte boundary (the swizzled x box);
          // a chunk that would straddle the end starts over at offset 0
          uint32_t off = hoff, pad = 0u;
          if (need) {
            off = (hoff + 1023u) & ~1023u;
            pad = off - hoff;
            if (off + need > (uint32_t)kRingBytes) {
              pad = (uint32_t)kRingBytes - hoff;
              off = 0u;
            }
          }
          const uint32_t start = head + pad;
          const bool full = start + need - tail > (uint32_t)kRingBytes || q - oldest >= (uint32_t)kRingSeq;
          if (full && !dep) resolve();   // releases need the pending x boxes
          // wait for the oldest chunks until the allocation fits and a barrier pair is free
          while (ok && (start + need - tail > (uint32_t)kRingBytes || q - oldest >= (uint32_t)kRingSeq)) {
            const uint32_t j = oldest % kRingSeq;
            if (!mbar_wait_bounded(&w_empty[j], (oldest / kRingSeq) & 1u, abort_flag, P.err, kDecWaitLimitNs,
                                   kDevErrTimeout)) {
              ok = false;
              break;
            }
            tail = w_end[j];
            ++oldest;
          }
          if (!ok) break;
          const uint32_t e = q % kRingSeq;
          w_off[e] = off;
          w_end[e] = start + need;
          head = start + need;
          hoff = off + need;
          uint8_t* dst = ring + off;
          fence_proxy_async_smem();
          mbar_arrive_expect_tx(&w_full[e], cnt ? bytes + xbytes : 0u);
          if (cnt) {
            if (dep) tma_load_3d(dst, &L.xmap, &w_full[e], 0, 0, (U.c0 + i) * (KW / 64));
            bulk_copy_g2s(dst + xbytes, L.tiles + (int64_t)m.x * KW, bytes, &w_full[e]);
          }
          if (!dep) ++n_pend;
        }
        if (!dep) resolve();
      }
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      q = __shfl_sync(0xffffffffu, q, 0);
      U = V;
      u = u_next;
      have = have_v;
    }
    if (lane == 0 && !ok) {
      // let copies already in flight land before the CTA retires
      for (uint32_t i = q > (uint32_t)kRingSeq ? q - kRingSeq : 0u; i < q; ++i) {
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait(&w_full[i % kRingSeq], (i / kRingSeq) & 1u))
          if (globaltimer_ns() - t0 > kDecDrainLimitNs) break;
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ consumer warps
    asm volatile("griddepcontrol.wait;" ::: "memory");
    // Warp pair (win, win + kDW) owns the 16-row window win: the first warp
    // takes a unit's even chunks, the second its odd chunks, so two chunks are
    // in the MMA pipeline per window.  At the unit's end one warp hands its
    // accumulator to the other through shared memory (the taker alternates
    // from unit to unit), which adds it and writes the result.
    const int win = warp & (kDW - 1), par = warp / kDW;
    const int g = lane >> 2, qd = lane & 3;
    const uint32_t lo_g = (1u << g) - 1u, lo_g8 = (1u << (g + 8)) - 1u;
    float* pbuf = pair_buf + win * (32 * 4 * kMaxNT) + lane * (4 * kMaxNT);
    uint32_t q = 0;
    bool ok = true;
    for (int k = 0; ok; ++k) {
      const int ms = k % kMetaSlots;
      if (!mbar_wait_bounded(&m_full[ms], (uint32_t)(k / kMetaSlots) & 1u, abort_flag, P.err, kDecWaitLimitNs,
                             kDevErrTimeout)) {
        ok = false;
        break;
      }
      const int u = unit_id[ms];
      if (u < 0) break;
      Unit U;
      unit_at(lay, P.n_layers, u, U);
      const DecLayer& L = P.L[U.l];
      const int4* mrow = meta + ms * kMaxCpu;
      float acc[NT][4], acc2[NT][4];   // two chains (even / odd k blocks) halve the MMA dependency depth
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[nt][i] = acc2[nt][i] = 0.f;
      for (int i = par; i < U.nC; i += 2) {
        const uint32_t qi = q + (uint32_t)i;   // ring sequence number of chunk i
        const int4 m = mrow[i];
        const uint32_t km = meta_mask(m, win);
        int base = 0;
#pragma unroll
        for (int w = 0; w < kDW; ++w)
          if (w < win) base += __popc(meta_mask(m, w));
        const int slot = (int)(qi % kRingSeq);
        if (!mbar_wait_bounded(&w_full[slot], (qi / kRingSeq) & 1u, abort_flag, P.err, kDecWaitLimitNs,
                               kDevErrTimeout)) {
          ok = false;
          break;
        }
        if (km != 0u) {
          const bool kg = (km >> g) & 1u, kg8 = (km >> (g + 8)) & 1u;
          const uint8_t* cbase = ring + w_off[slot];
          const uint4* sl = reinterpret_cast<const uint4*>(cbase + T * (2 * KW));
          const uint4* tg = sl + (base + __popc(km & lo_g)) * (KW / 8) + 2 * qd;
          const uint4* tg8 = sl + (base + __popc(km & lo_g8)) * (KW / 8) + 2 * qd;
#pragma unroll
          for (int b = 0; b < KW / 32; ++b) {
            const int j = 8 * (b >> 1) + (b & 1);
            const uint4 a = kg ? tg[j] : make_uint4(0u, 0u, 0u, 0u);
            const uint4 a8 = kg8 ? tg8[j] : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
              // x: slab s = b/2 holds k 64s..64s+63 of every token as 128-byte
              // rows (row index s*T + tok); 16-byte chunk c of a row sits at c ^ (row & 7)
              const int tok = nt * 8 + g;
              const int row = (b >> 1) * T + tok;
              const int ch = (2 * qd + (b & 1)) ^ (row & 7);
              const uint4 xv = tok < T ? *reinterpret_cast<const uint4*>(cbase + row * 128 + ch * 16)
                                       : make_uint4(0u, 0u, 0u, 0u);
              mma16816(acc[nt], a.x, a8.x, a.y, a8.y, xv.x, xv.y);
              mma16816(acc2[nt], a.z, a8.z, a.w, a8.w, xv.z, xv.w);
            }
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&w_empty[slot]);
      }
      q += (uint32_t)U.nC;
      if (!ok) break;
      __syncwarp();
      if (lane == 0) mbar_arrive(&m_empty[ms]);
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[nt][i] += acc2[nt][i];

      // ---- pair hand-off: one warp's accumulator joins the other's, which then
      // writes the unit's result; the writing role alternates between the two
      // warps from unit to unit, so the output path (and the split reduction's
      // global round trips) is shared evenly
      const uint32_t hpar = (uint32_t)k & 1u;
      if ((uint32_t)par != hpar) {
        if (!mbar_wait_bounded(&p_empty[win], hpar ^ 1u, abort_flag, P.err, kDecWaitLimitNs, kDevErrTimeout)) {
          ok = false;
          break;
        }
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
          *reinterpret_cast<float4*>(pbuf + 4 * nt) = make_float4(acc[nt][0], acc[nt][1], acc[nt][2], acc[nt][3]);
        __syncwarp();
        if (lane == 0) mbar_arrive(&p_full[win]);
        continue;
      }
      if (!mbar_wait_bounded(&p_full[win], hpar, abort_flag, P.err, kDecWaitLimitNs, kDevErrTimeout)) {
        ok = false;
        break;
      }
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const float4 o = *reinterpret_cast<const float4*>(pbuf + 4 * nt);
        acc[nt][0] += o.x;
        acc[nt][1] += o.y;
        acc[nt][2] += o.z;
        acc[nt][3] += o.w;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_empty[win]);

      // ---- unit result: this window's 16 rows x T tokens
      const int r0 = U.blk * kRows + win * kWin16;
      if (L.nsplit == 1) {
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
          for (int j = 0; j < 2; ++j) {
            const int tok = nt * 8 + 2 * qd + j;
            if (tok < T) {
              if (r0 + g < L.out) L.y[(int64_t)tok * L.out + r0 + g] = f32_to_bf16_rn(acc[nt][j]);
              if (r0 + g + 8 < L.out) L.y[(int64_t)tok * L.out + r0 + g + 8] = f32_to_bf16_rn(acc[nt][2 + j]);
            }
          }
      } else {
        const int split = U.c0 / L.cpu;
        float* part = L.ws + (((int64_t)U.blk * L.nsplit + split) * kDW + win) * kPartFloats;
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
          for (int j = 0; j < 2; ++j) {
            const int tok = nt * 8 + 2 * qd + j;
            part[tok * kWin16 + g] = acc[nt][j];
            part[tok * kWin16 + g + 8] = acc[nt][2 + j];
          }
        // The lanes' partial stores are ordered before lane 0's counter update
        // by the warp barrier; the update is an acquire-release RMW at GPU scope,
        // so it publishes them (release is cumulative), and in the last arriver
        // it acquires every other split's published partials, which the warp
        // barrier after the broadcast extends to all lanes (their loads go to L2).
        __syncwarp();
        int last = 0;
        int32_t* cnt = L.cnt + U.blk * kDW + win;
        if (lane == 0) last = (atom_add_acq_rel_gpu(cnt, 1) == L.nsplit - 1);
        last = __shfl_sync(0xffffffffu, last, 0);
        if (last) {
          __syncwarp();
          const float* base_ws = L.ws + ((int64_t)U.blk * L.nsplit * kDW + win) * kPartFloats;
          const int Tl = T < NT * 8 ? T : NT * 8;
          for (int e = lane; e < Tl * kWin16; e += 32) {
            // issue every partial's load first, then add them in split order
            float sum = 0.f;
            for (int s0 = 0; s0 < L.nsplit; s0 += 8) {
              float v[8];
#pragma unroll
              for (int u = 0; u < 8; ++u)
                v[u] = s0 + u < L.nsplit ? __ldcg(base_ws + (int64_t)(s0 + u) * kDW * kPartFloats + e) : 0.f;
#pragma unroll
              for (int u = 0; u < 8; ++u) sum += v[u];
            }
            const int tok = e / kWin16, i = e % kWin16;
            if (r0 + i < L.out) L.y[(int64_t)tok * L.out + r0 + i] = f32_to_bf16_rn(sum);
          }
          if (lane == 0) *cnt = 0;
        }
      }
    }
  }
  __syncthreads();
  // the last CTA to finish rewinds the ticket counter for the next launch
  if (threadIdx.x == 0) {
    __threadfence();
    if (atomicAdd(P.sched + 1, 1) == (int)gridDim.x - 1) {
      P.sched[0] = 0;
      P.sched[1] = 0;
      __threadfence();
    }
  }
}

// metadata of 64-row block b, chunk c: first packed row of the block's slice and
// the kept masks of its four 16-row windows
__global__ void k_pack_decode_meta(const int32_t* __restrict__ win_off16, const uint16_t* __restrict__ kmask16,
                              int32_t G, int32_t nw16, int32_t nblk, int4* __restrict__ dmeta) {
  const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;   // e = b * G + c
  if (e >= (int64_t)nblk * G) return;
  const int b = (int)(e / G), c = (int)(e % G);
  const int w0 = kDW * b;
  uint32_t km[kDW];
#pragma unroll
  for (int w = 0; w < kDW; ++w) km[w] = (w0 + w < nw16) ? kmask16[(int64_t)c * nw16 + w0 + w] : 0u;
  dmeta[e] = make_int4(win_off16[(int64_t)c * (nw16 + 1) + w0], (int)(km[0] | (km[1] << 16)),
                       (int)(km[2] | (km[3] << 16)), 0);
}

std::mutex g_slot_mu;

int sm_count_dec() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 148;
  }
  return n;
}

template <int NT, int MB, int KW>
cudaError_t launch_nt(const DecParams<MB>& P, int grid, cudaStream_t s) {
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(once, []() {
    attr_err = cudaFuncSetAttribute(k_decode<NT, MB, KW>, cudaFuncAttributeMaxDynamicSharedMemorySize, kDecSmemBytes);
  });
  if (attr_err != cudaSuccess) return attr_err;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kThreadsDec);
  cfg.dynamicSmemBytes = kDecSmemBytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k_decode<NT, MB, KW>, P);
}

}  // namespace

int decode_max_tokens() { return kMaxT; }

gs_status decode_prepare(gs_packed* p, cudaStream_t s) {
  p->nblk64 = (int32_t)((p->out + kRows - 1) / kRows);
  // Chunks per unit: a block's chunks are split into the whole number of
  // units nearest to its kept bytes / kUnitBytes (at most kMaxCpu chunks
  // each), of equal length.  Every split costs a partial write and a global
  // reduction, so a block only slightly above kUnitBytes stays whole instead
  // of leaving a one-chunk remainder unit.
  const double gbytes = 2.0 * (double)p->g_in;   // bytes of one kept group
  const double per_chunk = p->kept > 0 ? gbytes * (double)p->kept / ((double)p->G * (double)p->nblk64) : gbytes;
  int nsplit = (int)std::floor(per_chunk * (double)p->G / (double)kUnitBytes + 0.5);
  nsplit = std::min(p->G, std::max(nsplit, std::max(1, (p->G + kMaxCpu - 1) / kMaxCpu)));
  const int cpu = (p->G + nsplit - 1) / nsplit;
  p->dec_cpu = cpu;
  p->dec_cpu_fine = std::max(1, cpu / 4);
  p->dec_nsplit_max = (p->G + p->dec_cpu_fine - 1) / p->dec_cpu_fine;
  const size_t nmeta = (size_t)p->nblk64 * (size_t)p->G;
  {
    const gs_status am = lib_malloc(reinterpret_cast<void**>(&p->dmeta), nmeta * sizeof(int4));
    if (am != GS_OK) return am;
  }
  p->device_bytes += nmeta * sizeof(int4);
  // the split scratch of gs_pack's stream is made now (gs_linear on that
  // stream then never allocates); other streams get theirs on first use
  const DecSlot* slot = nullptr;
  const gs_status st = decode_slot(p, s, &slot);
  if (st != GS_OK) return st;
  const int64_t n = (int64_t)nmeta;
  k_pack_decode_meta<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(p->win_off16, p->kmask16, p->G, p->nw16, p->nblk64,
                                                           p->dmeta);
  note_launch();
  return cudaGetLastError() == cudaSuccess ? GS_OK : GS_ERR_CUDA;
}

void decode_release(gs_packed* p) {
  if (p->dmeta) cudaFree(p->dmeta);
  p->dmeta = nullptr;
  std::lock_guard<std::mutex> lk(g_slot_mu);
  for (int i = 0; i < p->dec_nslots; ++i) {
    if (p->dec_slot[i].ws) cudaFree(p->dec_slot[i].ws);
    if (p->dec_slot[i].cnt) cudaFree(p->dec_slot[i].cnt);
    p->dec_slot[i] = DecSlot{};
  }
  p->dec_nslots = 0;
}

gs_status decode_slot(const gs_packed* pc, cudaStream_t s, const DecSlot** out) {
  gs_packed* p = const_cast<gs_packed*>(pc);   // the slot table is the only mutable part of a handle
  const size_t nws = (size_t)p->nblk64 * p->dec_nsplit_max * kDW * kPartFloats;
  const size_t ncnt = (size_t)p->nblk64 * kDW + 2;   // + {unit ticket, finished CTAs}
  const uint64_t epoch = timeout_epoch();
  std::lock_guard<std::mutex> lk(g_slot_mu);
  DecSlot* slot = nullptr;
  for (int i = 0; i < p->dec_nslots; ++i)
    if (p->dec_slot[i].stream == static_cast<void*>(s)) slot = &p->dec_slot[i];
  if (!slot) {
    if (p->dec_nslots >= kDecSlots) return GS_ERR_UNSUPPORTED;
    DecSlot n{};
    n.stream = static_cast<void*>(s);
    // The stream may be capturing a CUDA graph (e.g. a capture side stream that
    // has not run a decode call before).  The slot is made outside the capture:
    // this thread's capture mode is relaxed while the buffers are allocated and
    // zeroed on a private non-blocking stream, then restored.
    cudaStreamCaptureMode mode = cudaStreamCaptureModeRelaxed;
    if (cudaThreadExchangeStreamCaptureMode(&mode) != cudaSuccess) return GS_ERR_CUDA;
    gs_status st = lib_malloc(reinterpret_cast<void**>(&n.ws), nws * sizeof(float));
    if (st == GS_OK) st = lib_malloc(reinterpret_cast<void**>(&n.cnt), ncnt * sizeof(int32_t));
    if (st == GS_OK) {
      cudaStream_t zs = nullptr;
      if (cudaStreamCreateWithFlags(&zs, cudaStreamNonBlocking) != cudaSuccess ||
          cudaMemsetAsync(n.cnt, 0, ncnt * sizeof(int32_t), zs) != cudaSuccess || cudaStreamSynchronize(zs) != cudaSuccess)
        st = GS_ERR_CUDA;
      if (zs) cudaStreamDestroy(zs);
    }
    cudaThreadExchangeStreamCaptureMode(&mode);
    if (st != GS_OK) {
      if (n.ws) cudaFree(n.ws);
      if (n.cnt) cudaFree(n.cnt);
      return st;
    }
    n.epoch = epoch;
    p->dec_slot[p->dec_nslots] = n;
    slot = &p->dec_slot[p->dec_nslots++];
    p->device_bytes += nws * sizeof(float) + ncnt * sizeof(int32_t);
  } else if (slot->epoch != epoch) {
    // a timed-out launch may have left arrival counters or the ticket half counted
    if (cudaMemsetAsync(slot->cnt, 0, ncnt * sizeof(int32_t), s) != cudaSuccess) return GS_ERR_CUDA;
    slot->epoch = epoch;
  }
  *out = slot;
  return GS_OK;
}

gs_status launch_decode(const gs_packed* const* ps, const void* const* xs, void* const* ys, int n, int T,
                        cudaStream_t s) {
  if (n <= 0 || T <= 0) return GS_OK;
  if (n > kMaxBatch || T > kMaxT) return GS_ERR_UNSUPPORTED;
  const int kw = ps[0]->g_in;   // one chunk width per launch
  for (int i = 1; i < n; ++i)
    if (ps[i]->g_in != kw) return GS_ERR_UNSUPPORTED;
  if (kw != 128 && kw != 256) return GS_ERR_UNSUPPORTED;
  // Unit list: layers in descending kept bytes.  Measured on the LLaMA-2-7B
  // block (per-module densities 0.3-0.7): every order that leaves the layer
  // whose blocks are split over several units (the down projection) at the end
  // loses about 12 % to its last-arriver reductions stretching the end of the
  // launch; big layers first keeps it early.  When the list would not give
  // every CTA a couple of units, all layers use quarter-size units (their split
  // reductions cost more than a ragged end does otherwise).
  std::vector<int> order(n);
  for (int i = 0; i < n; ++i) order[i] = i;
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return ps[a]->kept > ps[b]->kept; });
  const int64_t max_grid = 2 * (int64_t)sm_count_dec();
  int64_t coarse_units = 0;
  for (int i = 0; i < n; ++i) {
    const gs_packed* p = ps[i];
    coarse_units += (int64_t)p->nblk64 * ((p->G + p->dec_cpu - 1) / p->dec_cpu);
  }
  const bool all_fine = coarse_units < 2 * max_grid;
  std::vector<char> fine(n, all_fine ? 1 : 0);
  DecParams<kMaxBatch> P;
  std::memset(&P, 0, sizeof(P));
  P.n_layers = n;
  P.T = T;
  P.err = device_error_flag();
  if (!P.err) return GS_ERR_CUDA;
  int64_t units = 0;
  const DecSlot* first_slot = nullptr;
  for (int k = 0; k < n; ++k) {
    const gs_packed* p = ps[order[k]];
    DecLayer& L = P.L[k];
    const DecSlot* slot = nullptr;
    const gs_status st = decode_slot(p, s, &slot);
    if (st != GS_OK) return st;
    if (order[k] == 0) first_slot = slot;
    L.x = static_cast<const uint16_t*>(xs[order[k]]);
    if (!encode_tmap_slabs_bf16(&L.xmap, L.x, (uint64_t)p->in, (uint64_t)T, (uint32_t)T, (uint32_t)(kw / 64)))
      return GS_ERR_CUDA;
    L.tiles = p->tiles;
    L.dmeta = p->dmeta;
    L.y = static_cast<uint16_t*>(ys[order[k]]);
    L.ws = slot->ws;
    L.cnt = slot->cnt;
    L.out = (int32_t)p->out;
    L.in = (int32_t)p->in;
    L.G = p->G;
    L.nblk = p->nblk64;
    L.cpu = fine[k] ? p->dec_cpu_fine : p->dec_cpu;
    L.nsplit = (p->G + L.cpu - 1) / L.cpu;
    L.unit_begin = (int32_t)units;
    units += (int64_t)p->nblk64 * L.nsplit;
  }
  if (units > INT32_MAX) return GS_ERR_UNSUPPORTED;
  P.n_units = (int32_t)units;
  P.sched = first_slot->cnt + (size_t)ps[0]->nblk64 * kDW;
  P.inject_ns = take_injected_wait(GS_ALGO_DECODE);
  const int grid = (int)std::min<int64_t>(units, max_grid);
  cudaError_t e;
  if (n <= kSmallBatch) {
    DecParams<kSmallBatch> Q;
    std::memcpy(Q.L, P.L, sizeof(Q.L));
    Q.n_layers = P.n_layers;
    Q.T = P.T;
    Q.n_units = P.n_units;
    Q.sched = P.sched;
    Q.err = P.err;
    Q.inject_ns = P.inject_ns;
    if (kw == 256) e = T <= 8 ? launch_nt<1, kSmallBatch, 256>(Q, grid, s) : launch_nt<2, kSmallBatch, 256>(Q, grid, s);
    else e = T <= 8 ? launch_nt<1, kSmallBatch, 128>(Q, grid, s) : launch_nt<2, kSmallBatch, 128>(Q, grid, s);
  } else {
    if (kw == 256) e = T <= 8 ? launch_nt<1, kMaxBatch, 256>(P, grid, s) : launch_nt<2, kMaxBatch, 256>(P, grid, s);
    else e = T <= 8 ? launch_nt<1, kMaxBatch, 128>(P, grid, s) : launch_nt<2, kMaxBatch, 128>(P, grid, s);
  }
  note_launch();
  return e == cudaSuccess ? GS_OK : GS_ERR_CUDA;
}

}  // namespace gs
