// Device-side helpers shared by the kernels of libbdcommit: the vocabulary
// work plan, PTX wrappers for mbarriers, TMA, tcgen05 (UMMA + tensor memory),
// bounded waits and the online softmax combine.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>

namespace bd {

// Device status bits, OR-ed into the library's status word.
constexpr uint32_t DEV_TIMEOUT = 1u;
// A kernel found itself launched in a shape it cannot run (e.g. a CTA-pair
// kernel without its cluster of 2) and returned without doing anything.
constexpr uint32_t DEV_BAD_LAUNCH = 2u;

// A bounded wait gives up after this long (nanoseconds of %globaltimer).
constexpr uint64_t WAIT_LIMIT_NS = 1000000000ull;  // 1 s
// After giving up, drains of in-flight copies / MMAs wait at most this long.
constexpr uint64_t DRAIN_LIMIT_NS = 100000000ull;  // 0.1 s

constexpr float LOG2E = 1.4426950408889634f;
// The epilogues form the exponent of exp(l - m) as fmaf(l, log2 e, -mc) with
// mc = fl32(m log2 e): one instruction, but every exponent then carries mc's
// rounding error (up to half an ulp of m log2 e), which at the maximum itself
// should be 0. Below this magnitude of mc that error stays under 2^-13
// (relative error 1e-4 in the sum); states with a larger running max (logits
// beyond ~1400) form (l - m) log2 e instead, exact at l = m.
constexpr float FUSED_SHIFT_LIMIT = 2048.f;

// -------------------------------------------------------------------------
// Work plan of the LM-head kernels.
//
// The N compacted rows are cut into m-tiles of BM rows (token groups of the
// pair kernel) and the vocabulary into v-tiles of BN entries. A runner (a CTA,
// a CTA pair, or a cluster of pairs) holds MC consecutive m-tiles at once
// (the pair kernel's 4-CTA clusters: two CTA pairs, one m-tile each, sharing
// every head tile through multicast loads); "m-tiles" below count runner
// m-tiles of MC m-tiles (a missing last m-tile is computed on zero rows and
// written nowhere).
//
// The m-tiles are cut into bands of GM (the last band may be smaller) and the
// vocabulary into gv contiguous parts of (nearly) equal length (in steps of vc
// v-tiles when a runner takes vc at a time). A part of a band is the gm units
// (m-tile, part) that share the same head slice; a unit leaves one partial
// (max, sum of exponentials, argmax) per row and CTA (and pair, with vc = 2)
// in the slots of its part. Parts, ordered band by
// band, are packed whole into rounds of G units (G runners): a part that does
// not fit what is left of a round starts the next round, and runner c takes
// slot c of every round (a slot past the round's parts is idle). All m-tiles
// of a part therefore run at the same time, so its head slice is fetched from
// HBM once and re-read from L2 by the others; a part split across two rounds
// (an earlier round-robin plan) was fetched twice, a round apart.
//
// (GM, gv): among the pairs whose makespan rounds * (2 ceil(n_vt / gv) + 1)
// (in half v-tiles: half a v-tile for each unit's start and finish) is within
// 5% (MAKESPAN_SLACK_DIV) of the best, the fewest bands (each band streams the head
// once), then the smaller makespan, then the smaller gv; over GM <= min(n_mt,
// G) with GM m-tiles of rows within the in-flight budget below (they stay in
// L2 while their parts run) and gv <= min(G, n_vt). N is only known on the
// device: the compaction kernel evaluates the rule with one warp and stores
// the plan beside N in the workspace header (HDR_* below), which the LM-head
// and merge kernels read.
// -------------------------------------------------------------------------
struct BandPlan {
  int BM;         // rows per m-tile; 0 = derived from N (token groups of the pair kernel)
  int BN;         // vocabulary entries per v-tile
  int GM;         // m-tiles per band when > 0 (clamped to 1..n_mt); 0 = chosen with gv
  int G;          // runners that can run at once (CTAs, CTA pairs or clusters)
  int n_vt;       // ceil(V / BN)
  int cpu;        // CTAs per unit: each writes its own partial, so a part has cpu slots
  int vt_kb;      // KiB of head per v-tile (BN rows as the kernel reads them)
  int row_bytes;  // bytes of one packed token row as the kernel reads it
  int mc;         // m-tiles a runner holds at once (1, or 2 for 4-CTA clusters sharing head tiles)
  int vc;         // v-tiles a runner takes at once (1, or 2 for 4-CTA clusters sharing token rows)
  int gv_fixed;   // vocabulary parts when > 0 (clamped to 1..min(G, n_vt)), else chosen
  int rr;         // 1: units taken round-robin (runner c: units c, c + G, ...) instead of packed rounds
  int G2;         // spill runners: single CTA pairs on the SMs the clusters leave free (0: none)
  int spill_pct;  // a spill pair's time per tile against a cluster pair's, in percent (0: 100)
  int role;       // 0: the main launch; 1: the spill launch (single pairs, the last v-tiles)
};

// Words of the workspace header (int32) the kernel that learns N writes for
// the LM-head and merge kernels: N, the partial slots per row over all
// launches (parts times the CTAs that write a partial per unit), the main
// launch's band size and parts, the spill launch's band size and parts, the
// v-tile where the spill launch's range begins (n_vt without a spill launch)
// and the spill launch's first slot.
enum : int {
  HDR_N = 0, HDR_SLOTS = 1, HDR_GM = 2, HDR_GV = 3, HDR_GM2 = 4, HDR_GV2 = 5, HDR_VSPLIT = 6, HDR_SLOT0 = 7,
  HDR_WORDS = 8
};

__host__ __device__ __forceinline__ int cdiv(int a, int b) { return (a + b - 1) / b; }

// Token-group size of the pair kernel for N rows: the fewest groups of at most
// 256 rows, equal sizes rounded up to a multiple of 32 (16 rows per CTA).
__host__ __device__ __forceinline__ int pair_group_rows(int n_rows) {
  if (n_rows <= 0) return 32;
  const int groups = cdiv(n_rows, 256);
  return cdiv(cdiv(n_rows, groups), 32) * 32;
}

__host__ __device__ __forceinline__ int plan_bm(const BandPlan& p, int n_rows) {
  return p.BM > 0 ? p.BM : pair_group_rows(n_rows);
}

__host__ __device__ __forceinline__ int plan_mc(const BandPlan& p) { return p.mc > 1 ? p.mc : 1; }
__host__ __device__ __forceinline__ int plan_vc(const BandPlan& p) { return p.vc > 1 ? p.vc : 1; }

// Runner m-tiles (of plan_mc m-tiles each) for N rows; 0 without rows.
__host__ __device__ __forceinline__ int plan_runner_mts(const BandPlan& p, int n_rows) {
  return n_rows > 0 ? cdiv(cdiv(n_rows, plan_bm(p, n_rows)), plan_mc(p)) : 0;
}

// Rows of the m-tiles in flight (one band) are kept within ROWS_IN_FLIGHT
// bytes, or ROWS_IN_FLIGHT_MANY when there are more than two rounds' worth of
// m-tiles: over many rounds the runners drift apart, the units in flight span
// neighbouring bands, and larger bands no longer stay in L2 (the 256 x 8 x 64
// window read 134 GB with bands of 12 runner m-tiles, 52 GB with bands of 2).
constexpr int64_t ROWS_IN_FLIGHT = int64_t(64) << 20;
constexpr int64_t ROWS_IN_FLIGHT_MANY = int64_t(12) << 20;
// Among (GM, gv) within 1 + 1/MAKESPAN_SLACK_DIV (5%) of the best makespan,
// the fewest bands win. The plan's arithmetic is integer throughout: the
// kernel that learns N evaluates it on the device, where float64 is slow.
constexpr uint64_t MAKESPAN_SLACK_DIV = 20;

// The packing of the parts into rounds, for n_mt m-tiles, bands of gm and gv
// parts: nb full bands (their parts hold gm units, k1 per round) and, when
// rem > 0, a last band whose parts hold rem units (kr per round). The full
// bands' parts fill rounds 0..R0-1 and u0 units of round R0; f of the last
// band's parts share round R0 (when u0 > 0), the others follow kr per round.
struct Packing {
  int nb, rem, k1, kr, R0, u0, f, rounds;
};

__host__ __device__ __forceinline__ Packing plan_pack(int n_mt, int G, int gm, int gv) {
  Packing k;
  k.nb = n_mt / gm;
  k.rem = n_mt - k.nb * gm;
  k.k1 = G / gm;
  k.kr = k.rem > 0 ? G / k.rem : 0;
  // nb * gv < 2^28 (at most 2^19 m-tiles of 2^24 positions, gv <= 304): 32-bit
  const int full_parts = k.nb * gv;
  k.R0 = full_parts / k.k1;
  k.u0 = (full_parts - k.R0 * k.k1) * gm;
  int left = k.rem > 0 ? gv : 0;
  k.f = 0;
  if (k.u0 > 0 && k.rem > 0) {
    const int fit = (G - k.u0) / k.rem;
    k.f = fit < left ? fit : left;
  }
  left -= k.f;
  k.rounds = k.R0 + (k.u0 > 0 ? 1 : 0) + (left > 0 ? cdiv(left, k.kr) : 0);
  return k;
}

// The makespan of (gm, gv) in half v-tiles (saturated at 2^33 - 1).
__host__ __device__ __forceinline__ uint64_t plan_cost(const BandPlan& p, int n_mt, int gm, int gv) {
  const Packing k = plan_pack(n_mt, p.G, gm, gv);
  const uint64_t cost = static_cast<uint64_t>(k.rounds) * (2 * static_cast<uint64_t>(cdiv(p.n_vt, gv)) + 1);
  return cost < (uint64_t(1) << 33) ? cost : (uint64_t(1) << 33) - 1;
}

// The choice key of (gm, gv) among those within the slack: bands, then
// makespan, then gv (smallest wins), gm in the low bits for decoding.
__host__ __device__ __forceinline__ uint64_t plan_key(const BandPlan& p, int n_mt, int gm, int gv, uint64_t cost) {
  uint64_t nbands = static_cast<uint64_t>(cdiv(n_mt, gm));
  if (nbands > 1023) nbands = 1023;
  return (nbands << 53) | (cost << 20) | (static_cast<uint64_t>(gv) << 10) | static_cast<uint64_t>(gm);
}

// The range of band sizes the choice may take: GM if fixed; else 1..min(n_mt,
// G) limited to ROWS_IN_FLIGHT of rows (at least 1).
__host__ __device__ __forceinline__ void plan_gm_range(const BandPlan& p, int bm, int n_mt, int* lo, int* hi) {
  const int top = n_mt < p.G ? n_mt : p.G;
  if (p.GM > 0) {
    *lo = *hi = p.GM < top ? p.GM : (top > 0 ? top : 1);
    return;
  }
  const int64_t tile = static_cast<int64_t>(bm) * plan_mc(p) * (p.row_bytes > 0 ? p.row_bytes : 1);
  int cap = static_cast<int>((n_mt > 2 * p.G ? ROWS_IN_FLIGHT_MANY : ROWS_IN_FLIGHT) / tile);
  if (cap < 1) cap = 1;
  *lo = 1;
  *hi = top < cap ? top : cap;
  if (*hi < 1) *hi = 1;
}

__host__ __device__ __forceinline__ void plan_gv_range(const BandPlan& p, int* lo, int* hi) {
  const int top = p.G < p.n_vt ? p.G : p.n_vt;
  if (p.gv_fixed > 0) {
    *lo = *hi = p.gv_fixed < top ? p.gv_fixed : top;
  } else {
    *lo = 1;
    *hi = top;
  }
}

// (GM, gv) for n_mt runner m-tiles, sequentially (host).
__host__ __device__ __forceinline__ void plan_choose(const BandPlan& p, int n_rows, int* gm_out, int* gv_out) {
  const int n_mt = plan_runner_mts(p, n_rows) > 0 ? plan_runner_mts(p, n_rows) : 1;
  int glo, ghi, vlo, vhi;
  plan_gm_range(p, plan_bm(p, n_rows), n_mt, &glo, &ghi);
  plan_gv_range(p, &vlo, &vhi);
  uint64_t c_min = ~uint64_t(0);
  for (int gm = glo; gm <= ghi; ++gm)
    for (int gv = vlo; gv <= vhi; ++gv) {
      const uint64_t c = plan_cost(p, n_mt, gm, gv);
      c_min = c < c_min ? c : c_min;
    }
  const uint64_t c_max = c_min + c_min / MAKESPAN_SLACK_DIV;
  uint64_t best = ~uint64_t(0);
  for (int gm = glo; gm <= ghi; ++gm)
    for (int gv = vlo; gv <= vhi; ++gv) {
      const uint64_t c = plan_cost(p, n_mt, gm, gv);
      if (c > c_max) continue;
      const uint64_t k = plan_key(p, n_mt, gm, gv, c);
      best = k < best ? k : best;
    }
  *gm_out = static_cast<int>(best & 1023u);
  *gv_out = static_cast<int>((best >> 10) & 1023u);
}

#ifdef __CUDACC__
// The same choice by a whole warp, 32 candidates at a time (the kernel that
// learns N calls it once and stores GM and gv in the workspace header).
__device__ __forceinline__ void plan_choose_warp(const BandPlan& p, int n_rows, int* gm_out, int* gv_out) {
  const int n_mt = plan_runner_mts(p, n_rows) > 0 ? plan_runner_mts(p, n_rows) : 1;
  int glo, ghi, vlo, vhi;
  plan_gm_range(p, plan_bm(p, n_rows), n_mt, &glo, &ghi);
  plan_gv_range(p, &vlo, &vhi);
  const int nv = vhi - vlo + 1;
  const int total = (ghi - glo + 1) * nv;
  const int lane = static_cast<int>(threadIdx.x & 31);
  // the first 32 * CACHED candidates' costs stay in registers for the second pass
  constexpr int CACHED = 4;
  uint64_t cc[CACHED];
  uint64_t c_min = ~uint64_t(0);
#pragma unroll
  for (int q = 0; q < CACHED; ++q) {
    const int i = lane + 32 * q;
    cc[q] = i < total ? plan_cost(p, n_mt, glo + i / nv, vlo + i % nv) : ~uint64_t(0);
    c_min = cc[q] < c_min ? cc[q] : c_min;
  }
  for (int i = lane + 32 * CACHED; i < total; i += 32) {
    const uint64_t c = plan_cost(p, n_mt, glo + i / nv, vlo + i % nv);
    c_min = c < c_min ? c : c_min;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const uint64_t other = __shfl_xor_sync(0xffffffffu, c_min, o);
    c_min = other < c_min ? other : c_min;
  }
  const uint64_t c_max = c_min + c_min / MAKESPAN_SLACK_DIV;
  uint64_t best = ~uint64_t(0);
#pragma unroll
  for (int q = 0; q < CACHED; ++q) {
    const int i = lane + 32 * q;
    if (i < total && cc[q] <= c_max) {
      const uint64_t k = plan_key(p, n_mt, glo + i / nv, vlo + i % nv, cc[q]);
      best = k < best ? k : best;
    }
  }
  for (int i = lane + 32 * CACHED; i < total; i += 32) {
    const uint64_t c = plan_cost(p, n_mt, glo + i / nv, vlo + i % nv);
    if (c > c_max) continue;
    const uint64_t k = plan_key(p, n_mt, glo + i / nv, vlo + i % nv, c);
    best = k < best ? k : best;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const uint64_t other = __shfl_xor_sync(0xffffffffu, best, o);
    best = other < best ? other : best;
  }
  *gm_out = static_cast<int>(best & 1023u);
  *gv_out = static_cast<int>((best >> 10) & 1023u);
}
#endif

// Spill runners. Clusters of two CTA pairs cannot fill every SM (152 SMs hold
// 36 clusters of 4 CTAs); the G2 pairs that still fit run as a second,
// concurrent launch of single pairs (role 1) over the last v-tiles. The
// vocabulary is split so that both launches carry the same time per pair:
// the main launch's G runners take n_rmt runner m-tiles (mc m-tiles each) of
// vsplit v-tiles, vc at a time (one per pair either way), the spill pairs n_mt
// m-tiles of the remaining n_vt - vsplit v-tiles at spill_pct percent of a
// cluster pair's time per tile. With vc = 2 vsplit is even, so the main
// launch's v-tile pairs stay in its range. Each launch then chooses its own
// (GM, gv) over its own range.
__host__ __device__ __forceinline__ int plan_vsplit(const BandPlan& p, int n_rows) {
  if (p.G2 <= 0 || n_rows <= 0) return p.n_vt;
  const int64_t n_mt = cdiv(n_rows, plan_bm(p, n_rows));
  const int64_t n_rmt = plan_runner_mts(p, n_rows);
  const int64_t vc = plan_vc(p);
  const int64_t pct = p.spill_pct > 0 ? p.spill_pct : 100;
  // n_rmt vsplit / (G vc) = (pct / 100) n_mt (n_vt - vsplit) / G2, rounded to nearest
  const int64_t num = pct * n_mt * p.n_vt * p.G * vc;
  const int64_t den = 100 * n_rmt * p.G2 + pct * n_mt * p.G * vc;
  int vsplit = static_cast<int>((2 * num + den) / (2 * den));
  if (vc == 2) vsplit &= ~1;
  if (vsplit < static_cast<int>(vc)) vsplit = static_cast<int>(vc);
  if (vsplit > p.n_vt - static_cast<int>(vc)) vsplit = p.n_vt;  // nothing left for the spill launch
  return vsplit;
}

// Partial slots a unit writes per row: its CTAs' partials (a CTA pair writes
// one per CTA; with vc = 2 each pair of the cluster writes its own).
__host__ __device__ __forceinline__ int plan_unit_slots(const BandPlan& p) { return p.cpu * plan_vc(p); }
constexpr int SPILL_UNIT_SLOTS = 2;  // a single CTA pair

// The plan of one launch over its share of the vocabulary (role 0: v-tiles
// [0, vsplit), in steps of vc; role 1: [vsplit, n_vt)). n_vt of the result
// counts the launch's steps.
__host__ __device__ __forceinline__ BandPlan plan_share(const BandPlan& p, int vsplit, int role) {
  BandPlan q = p;
  q.role = role;
  if (role == 0) {
    q.n_vt = cdiv(vsplit, plan_vc(p));
  } else {
    q.n_vt = p.n_vt - vsplit;
    q.G = p.G2;
    q.mc = 1;
    q.vc = 1;
    q.cpu = SPILL_UNIT_SLOTS;
    q.GM = 0;
    q.gv_fixed = 0;
  }
  return q;
}

// The header words from the two launches' choices.
__host__ __device__ __forceinline__ void plan_fill_header(const BandPlan& p, int n_rows, int vsplit, int gm, int gv,
                                                          int gm2, int gv2, int* hdr) {
  hdr[HDR_N] = n_rows;
  hdr[HDR_SLOTS] = gv * plan_unit_slots(p) + gv2 * SPILL_UNIT_SLOTS;
  hdr[HDR_GM] = gm;
  hdr[HDR_GV] = gv;
  hdr[HDR_GM2] = gm2;
  hdr[HDR_GV2] = gv2;
  hdr[HDR_VSPLIT] = vsplit;
  hdr[HDR_SLOT0] = gv * plan_unit_slots(p);
}

// The workspace header for N rows, sequentially (host).
__host__ __device__ __forceinline__ void plan_header(const BandPlan& p, int n_rows, int* hdr) {
  const int vsplit = plan_vsplit(p, n_rows);
  int gm = 1, gv = 1, gm2 = 0, gv2 = 0;
  plan_choose(plan_share(p, vsplit, 0), n_rows, &gm, &gv);
  if (vsplit < p.n_vt) plan_choose(plan_share(p, vsplit, 1), n_rows, &gm2, &gv2);
  plan_fill_header(p, n_rows, vsplit, gm, gv, gm2, gv2, hdr);
}

#ifdef __CUDACC__
// The same header by one warp (the kernel that learns N calls it once); lane
// 0 writes it.
__device__ __forceinline__ void plan_write_header(const BandPlan& p, int n_rows, int* hdr) {
  const int vsplit = plan_vsplit(p, n_rows);
  int gm = 1, gv = 1, gm2 = 0, gv2 = 0;
  plan_choose_warp(plan_share(p, vsplit, 0), n_rows, &gm, &gv);
  if (vsplit < p.n_vt) plan_choose_warp(plan_share(p, vsplit, 1), n_rows, &gm2, &gv2);
  if ((threadIdx.x & 31) == 0) plan_fill_header(p, n_rows, vsplit, gm, gv, gm2, gv2, hdr);
}
#endif

// A header word, read past L1: the spill launch starts without waiting on
// the kernel that wrote the header (that kernel has completed by then).
__host__ __device__ __forceinline__ int hdr_word(const int* hdr, int i) {
#ifdef __CUDA_ARCH__
  return __ldcg(hdr + i);
#else
  return hdr[i];
#endif
}

// Partial slots per row the arrays hold at most, over both launches.
__host__ __device__ __forceinline__ int plan_max_slots(const BandPlan& p) {
  const int steps = cdiv(p.n_vt, plan_vc(p));
  int s = plan_unit_slots(p) * (p.G < steps ? p.G : steps);
  if (p.G2 > 0) s += SPILL_UNIT_SLOTS * (p.G2 < p.n_vt ? p.G2 : p.n_vt);
  return s;
}

// Iterates the units of runner `runner` under the packed plan.
struct TileIter {
  int runner, G;
  int n_mt, gm, gv, n_vt, mc, rr;
  int vt0;     // first v-tile of this launch's range
  int slot0;   // partial slots of the other launch before this one's
  Packing k;
  int round;
  int m_tile;  // current m-tile (the first of the runner's mc m-tiles)
  int part;    // vocabulary part of the current unit (this launch's)
  int vt, vt_end;  // its range in steps of vc v-tiles (the spill launch: v-tiles from vt0)

  // hdr: the workspace header the kernel that learns N wrote (HDR_*)
  __host__ __device__ void init(const BandPlan& plan, const int* hdr, int runner_index) {
    runner = runner_index;
    G = plan.G;
    mc = plan_mc(plan);
    const int n_rows = hdr_word(hdr, HDR_N);
    n_mt = plan_runner_mts(plan, n_rows);
    const bool spill = plan.role == 1;
    const int vsplit = hdr_word(hdr, HDR_VSPLIT);
    gm = hdr_word(hdr, spill ? HDR_GM2 : HDR_GM);
    gv = hdr_word(hdr, spill ? HDR_GV2 : HDR_GV);
    vt0 = spill ? vsplit : 0;
    n_vt = spill ? plan.n_vt - vsplit : cdiv(vsplit, plan_vc(plan));  // steps of vc v-tiles
    slot0 = spill ? hdr_word(hdr, HDR_SLOT0) : 0;
    if (gm < 1) gm = 1;
    const bool none = n_mt == 0 || gv < 1 || n_vt < 1;
    if (gv < 1) gv = 1;
    k = plan_pack(n_mt > 0 ? n_mt : 1, G, gm, gv);
    rr = plan.rr;
    if (rr) k.rounds = static_cast<int>((static_cast<int64_t>(n_mt) * gv + G - 1) / G);
    if (none) k.rounds = 0;
    round = -1;
    vt = vt_end = 0;
  }
#ifdef __CUDACC__
  __device__ void init(const BandPlan& plan, const int* hdr) { init(plan, hdr, blockIdx.x); }
#endif
  // Round-robin order (plan.rr): unit u = c + r G in band-major, part-major
  // order; false past the last unit.
  __host__ __device__ bool unit_rr(int r) {
    const int64_t u = static_cast<int64_t>(r) * G + runner;
    if (u >= static_cast<int64_t>(n_mt) * gv) return false;
    const int64_t band_units = static_cast<int64_t>(gm) * gv;
    const int b = static_cast<int>(u / band_units);
    const int i = static_cast<int>(u - b * band_units);
    const int m0 = b * gm;
    const int g = n_mt - m0 < gm ? n_mt - m0 : gm;
    part = i / g;
    m_tile = (m0 + i % g) * mc;
    vt = vt0 + static_cast<int>(static_cast<int64_t>(part) * n_vt / gv);
    vt_end = vt0 + static_cast<int>(static_cast<int64_t>(part + 1) * n_vt / gv);
    return true;
  }
  // This runner's unit of round r: false if its slot is idle there.
  __host__ __device__ bool unit_of(int r) {
    if (rr) return unit_rr(r);
    const int c = runner;
    int64_t q = -1;  // part index in the global order (full bands first)
    int mt = 0;
    if (r < k.R0 || (r == k.R0 && c < k.u0)) {
      if (c >= k.k1 * gm) return false;
      q = static_cast<int64_t>(r) * k.k1 + c / gm;
      if (q >= static_cast<int64_t>(k.nb) * gv) return false;
      mt = static_cast<int>(q / gv) * gm + c % gm;
      part = static_cast<int>(q % gv);
    } else {
      if (k.rem == 0) return false;
      int j;  // part of the last band
      if (r == k.R0 && k.u0 > 0) {
        j = (c - k.u0) / k.rem;
        if (j >= k.f) return false;
        mt = k.nb * gm + (c - k.u0) % k.rem;
      } else {
        const int r2 = r - k.R0 - (k.u0 > 0 ? 1 : 0);
        if (c >= k.kr * k.rem) return false;
        j = k.f + r2 * k.kr + c / k.rem;
        if (j >= gv) return false;
        mt = k.nb * gm + c % k.rem;
      }
      part = j;
    }
    m_tile = mt * mc;
    vt = vt0 + static_cast<int>(static_cast<int64_t>(part) * n_vt / gv);
    vt_end = vt0 + static_cast<int>(static_cast<int64_t>(part + 1) * n_vt / gv);
    return true;
  }
  // Advances to the next unit; false when there is no more work.
  __host__ __device__ bool next_unit() {
    while (++round < k.rounds)
      if (unit_of(round)) return true;
    return false;
  }
};

// -------------------------------------------------------------------------
// Online softmax state: running max m (natural units), sum s of exp(l - m),
// lowest index a attaining m. Combine is commutative and keeps the lowest
// index on equal maxima.
// -------------------------------------------------------------------------
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ void softmax_combine(float& m, float& s, int& a, float m2, float s2, int a2) {
  if (m2 > m) {
    s = s2 + (m == -INFINITY ? 0.f : s * ex2_approx((m - m2) * LOG2E));
    m = m2;
    a = a2;
  } else if (m2 == m) {
    if (m2 != -INFINITY) s += s2;
    a = a2 < a ? a2 : a;
  } else if (m2 != -INFINITY) {
    s += s2 * ex2_approx((m2 - m) * LOG2E);
  }
}

// The same combine carrying t = sum exp(l - m) * (l - m) * log2(e), the first
// moment of the shifted logits in log2 units (the entropy accumulator of the
// verification path: H = ln s - t / (s * log2(e))). Rescaling a state from max
// m to M > m multiplies both sums by f = 2^((m - M) log2 e) and shifts every
// (l - m) by (m - M): t -> f * (t + (m - M) log2(e) * s).
__device__ __forceinline__ void softmax_combine_t(float& m, float& s, int& a, float& t, float m2, float s2, int a2,
                                                  float t2) {
  if (m2 > m) {
    if (m == -INFINITY) {
      t = t2;
      s = s2;
    } else {
      const float dm = (m - m2) * LOG2E;
      const float f = ex2_approx(dm);
      t = t2 + f * fmaf(dm, s, t);
      s = s2 + f * s;
    }
    m = m2;
    a = a2;
  } else if (m2 == m) {
    if (m2 != -INFINITY) {
      s += s2;
      t += t2;
    }
    a = a2 < a ? a2 : a;
  } else if (m2 != -INFINITY) {
    const float dm = (m2 - m) * LOG2E;
    const float f = ex2_approx(dm);
    t += f * fmaf(dm, s2, t2);
    s += f * s2;
  }
}

// -------------------------------------------------------------------------
// PTX wrappers
// -------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

// CLUSTER: acquire at cluster scope, for phases completed by arrivals that
// release writes made in the peer CTA's shared memory.
template <bool CLUSTER = false>
__device__ __forceinline__ uint32_t mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  if constexpr (CLUSTER) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
  } else {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
  }
  return ok;
}

// Single-thread bounded wait for the phase of parity `parity` to complete.
// Returns false (and raises the CTA's abort flag) after WAIT_LIMIT_NS, or as
// soon as another role of the CTA has raised the abort flag.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                          uint32_t* status) {
  if (mbar_try_wait(bar, parity)) return true;
  uint64_t t0 = globaltimer_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 31u) == 0) {
      if (*abort_flag) return false;
      if (globaltimer_ns() - t0 > WAIT_LIMIT_NS) {
        *abort_flag = 1;
        atomicOr(status, DEV_TIMEOUT);
        return false;
      }
    }
  }
}

// Whole-warp bounded wait with a warp-uniform outcome.
template <bool CLUSTER = false>
__device__ __forceinline__ bool mbar_wait_warp(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                               uint32_t* status) {
  const uint32_t lane = threadIdx.x & 31u;
  uint64_t t0 = 0;
  for (uint32_t it = 0;; ++it) {
    uint32_t ok = mbar_try_wait<CLUSTER>(bar, parity);
    if (__all_sync(0xffffffffu, ok)) return true;
    if ((it & 31u) == 31u) {
      int stop = 0;
      if (lane == 0) {
        uint64_t now = globaltimer_ns();
        if (t0 == 0) t0 = now;
        if (*abort_flag) {
          stop = 1;
        } else if (now - t0 > WAIT_LIMIT_NS) {
          *abort_flag = 1;
          atomicOr(status, DEV_TIMEOUT);
          stop = 1;
        }
      }
      if (__shfl_sync(0xffffffffu, stop, 0)) return false;
    }
  }
}

// Orders this thread's generic-proxy writes to shared memory before later
// async-proxy accesses (TMA, tcgen05.mma operand reads) of the same memory.
__device__ __forceinline__ void fence_proxy_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

__device__ __forceinline__ uint4 ld_shared_v4(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
  return v;
}

__device__ __forceinline__ uint32_t ld_shared_u16(uint32_t addr) {
  uint16_t v;
  asm volatile("ld.shared.u16 %0, [%1];" : "=h"(v) : "r"(addr));
  return v;
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}

// Two E2M1 codes (low nibble: the lower element) -> f16x2 (lower element in the low half); exact.
__device__ __forceinline__ uint32_t e2m1x2_to_f16x2(uint32_t byte) {
  uint32_t h2;
  asm("{\n\t.reg .b8 t;\n\tcvt.u8.u32 t, %1;\n\tcvt.rn.f16x2.e2m1x2 %0, t;\n\t}" : "=r"(h2) : "r"(byte));
  return h2;
}

// Two E4M3 values (low byte: the lower element) -> f16x2; exact (every E4M3 value is an f16).
__device__ __forceinline__ uint32_t e4m3x2_to_f16x2(uint32_t two) {
  uint32_t h2;
  asm("{\n\t.reg .b16 t;\n\tcvt.u16.u32 t, %1;\n\tcvt.rn.f16x2.e4m3x2 %0, t;\n\t}" : "=r"(h2) : "r"(two));
  return h2;
}

// f16x2 -> bf16x2 through fp32; exact for the values the head decodes produce
// (at most six significant bits, magnitudes between 2^-10 and 2688, or zero).
__device__ __forceinline__ uint32_t f16x2_to_bf16x2(uint32_t h2) {
  const __half2 h = *reinterpret_cast<const __half2*>(&h2);
  const float2 f = __half22float2(h);
  const __nv_bfloat162 b = __floats2bfloat162_rn(f.x, f.y);
  return *reinterpret_cast<const uint32_t*>(&b);
}

__device__ __forceinline__ uint32_t hmul2_u32(uint32_t a, uint32_t b) {
  const __half2 r = __hmul2(*reinterpret_cast<const __half2*>(&a), *reinterpret_cast<const __half2*>(&b));
  return *reinterpret_cast<const uint32_t*>(&r);
}

// True in exactly one lane of a converged warp (elect.sync). A role that
// issues asynchronous work (TMA copies, MMAs, commits) runs its loop in the
// whole warp, with warp-uniform barrier waits, and lets the elected lane
// issue: a single divergent lane that waits and issues pays a much larger
// per-instruction issue cost.
__device__ __forceinline__ bool elect_one() {
  uint32_t pred;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "elect.sync _|p, 0xffffffff;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(pred));
  return pred != 0;
}

// Bounded wait that ignores the abort flag (used only to drain work in flight
// before the CTA exits).
__device__ __forceinline__ bool mbar_drain(uint32_t bar, uint32_t parity) {
  uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer_ns() - t0 > DRAIN_LIMIT_NS) return false;
  }
  return true;
}

// ---- TMA ----------------------------------------------------------------
__device__ __forceinline__ void prefetch_tmap(const void* tmap) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tmap)) : "memory");
}

__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

__device__ __forceinline__ uint64_t policy_evict_normal() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(p));
  return p;
}

__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// L2 eviction priority of a stream of TMA loads: L2_EVICT_FIRST, L2_EVICT_NORMAL
// or L2_EVICT_LAST (the LM-head kernels take theirs from TcArgs).
enum : int { L2_EVICT_FIRST = 0, L2_EVICT_NORMAL = 1, L2_EVICT_LAST = 2 };
__device__ __forceinline__ uint64_t l2_policy(int sel) {
  return sel == L2_EVICT_LAST ? policy_evict_last() : sel == L2_EVICT_NORMAL ? policy_evict_normal() : policy_evict_first();
}

// 2-D tiled load global -> shared; completes `bytes` of transaction count on `bar`.
// x is the innermost (contiguous) coordinate in elements, y the row.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const void* tmap, uint32_t bar, int x, int y,
                                            uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(x), "r"(y), "r"(bar), "l"(policy)
      : "memory");
}

// ---- tcgen05 ------------------------------------------------------------
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
}

__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// Shared-memory matrix descriptor of a K-major operand tile stored with the
// 128-byte swizzle (rows of 64 bf16 = 128 B, 8-row swizzle atoms of 1 KB):
// start address >> 4 in bits 0-13, leading byte offset >> 4 in bits 16-29
// (unused for swizzled K-major layouts), stride byte offset >> 4 (1 KB
// between 8-row groups) in bits 32-45, descriptor version 1 in bits 46-47,
// base offset 0 (tiles are 1 KB aligned), swizzle mode 2 (128 B) in bits 61-63.
__device__ __forceinline__ uint64_t sw128_kmajor_desc(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>(16u >> 4) << 16;
  d |= static_cast<uint64_t>(1024u >> 4) << 32;
  d |= static_cast<uint64_t>(1u) << 46;
  d |= static_cast<uint64_t>(2u) << 61;
  return d;
}

// Instruction descriptor of tcgen05.mma kind::f16 with bf16 A and B, fp32
// accumulator, both operands K-major: D format F32 (bits 4-5 = 1), A format
// BF16 (bits 7-9 = 1), B format BF16 (bits 10-12 = 1), N >> 3 in bits 17-22,
// M >> 4 in bits 24-28.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(N >> 3) << 17) |
         (static_cast<uint32_t>(M >> 4) << 24);
}

// The same with f16 A and B (format code 0 in bits 7-9 and 10-12).
__host__ __device__ constexpr uint32_t idesc_f16_f32(int M, int N) {
  return (1u << 4) | (static_cast<uint32_t>(N >> 3) << 17) | (static_cast<uint32_t>(M >> 4) << 24);
}

// Instruction descriptor of tcgen05.mma kind::f8f6f4 with E4M3 A and B
// (format code 0 in bits 7-9 and 10-12), fp32 accumulator, both operands
// K-major; N >> 3 in bits 17-22, M >> 4 in bits 24-28.
__host__ __device__ constexpr uint32_t idesc_e4m3_f32(int M, int N) {
  return (1u << 4) | (static_cast<uint32_t>(N >> 3) << 17) | (static_cast<uint32_t>(M >> 4) << 24);
}

// D[tmem] (+)= A[smem] * B[smem]^T, issued by one thread.
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive once on `bar` when every tcgen05.mma issued so far by this thread has completed.
__device__ __forceinline__ void umma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}

// Load 32 consecutive fp32 columns of this thread's TMEM lane (32x32b shape,
// x32 repeat) and wait for the load to complete.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
        "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
        "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
        "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// ---- programmatic dependent launch ------------------------------------------
// Blocks until the grid this one depends on has completed and its writes are
// visible (a no-op when the launch carries no programmatic dependency).
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
// Lets the dependent grid be scheduled once every CTA of this grid has called
// it (or exited).
__device__ __forceinline__ void griddep_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// ---- clusters and the CTA pair (cta_group::2) ----------------------------
__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_nctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
  return r;
}

// All threads of both CTAs of the cluster.
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Shared::cluster address of the variable at CTA-local address `addr` in CTA `rank`.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}

// Arrive once on an mbarrier given by its shared::cluster address (possibly in the peer CTA).
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}

// 2-D tiled load into this CTA's shared memory whose completion is counted on
// an mbarrier of either CTA of the pair (`mbar` is a shared::cluster address).
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const void* tmap, uint32_t mbar, int x, int y,
                                                 uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.cta_group::2.L2::cache_hint"
      " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(x), "r"(y), "r"(mbar), "l"(policy)
      : "memory");
}

// The same load multicast to the CTAs of `cta_mask` (same CTA-relative
// address in each); each destination's bytes are counted on the mbarrier at
// mbar's offset in that destination's pair-issuing (even) CTA.
__device__ __forceinline__ void tma_load_2d_pair_mc(uint32_t dst, const void* tmap, uint32_t mbar, int x, int y,
                                                    uint16_t cta_mask, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.multicast::cluster.cta_group::2"
      ".L2::cache_hint [%0], [%1, {%2, %3}], [%4], %5, %6;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(x), "r"(y), "r"(mbar), "h"(cta_mask), "l"(policy)
      : "memory");
}

// Tensor memory of a CTA pair: one warp of each CTA executes these together.
__device__ __forceinline__ void tmem_alloc_pair(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
}

__device__ __forceinline__ void tmem_relinquish_pair() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

// D[tmem of both CTAs] (+)= A[smem of both CTAs] * B[smem of both CTAs]^T with
// M = 256 (128 rows of A in each CTA) and B's N rows split in halves between
// the CTAs; issued by one thread of the even CTA.
__device__ __forceinline__ void umma_bf16_pair(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                               uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// The same on a CTA pair with 8-bit operands (K = 32 per instruction).
__device__ __forceinline__ void umma_f8_pair(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                             uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive once on the mbarrier at CTA-local address `bar` in every CTA of
// `cta_mask` when all pair MMAs issued so far by this thread have completed.
__device__ __forceinline__ void umma_commit_pair_mc(uint32_t bar, uint16_t cta_mask) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(bar),
      "h"(cta_mask)
      : "memory");
}

__device__ __forceinline__ void named_barrier_sync(uint32_t id, uint32_t nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

}  // namespace bd
