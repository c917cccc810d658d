// Host check of the LM-head work plan (common.cuh): for each case given on
// the command line as "n_rows BM GM vt_kb row_bytes G n_vt cpu mc vc G2 spill_pct",
// the header the compaction kernel would write is formed, and over both
// launches (the main one and, with G2 > 0, the spill launch of G2 single
// pairs over the last v-tiles) every (m-tile, v-tile) pair is taken by
// exactly one unit (a runner holds mc m-tiles and takes vc v-tiles per step;
// a step's second v-tile past the vocabulary is computed and discarded), the
// units of every part run in the same round of their launch, the partial
// slots of the two launches do not overlap and stay below the slots the merge
// reads, and the busiest runner's steps are reported against the even share.
// Prints one line per case:
//   ok <n_mt> <gv> <slots> <max_steps> <ideal_time> <gm> <vsplit> <max_vtiles_spill> <gm2> <gv2>
//   or FAIL <reason>
#include <cstdio>
#include <cstdlib>
#include <vector>

#include "common.cuh"

int main(int argc, char** argv) {
  constexpr int NA = 12;
  for (int i = 1; i + NA - 1 < argc; i += NA) {
    bd::BandPlan p{};
    const int n_rows = std::atoi(argv[i]);
    p.BM = std::atoi(argv[i + 1]);
    p.GM = std::atoi(argv[i + 2]);
    p.vt_kb = std::atoi(argv[i + 3]);
    p.row_bytes = std::atoi(argv[i + 4]);
    p.G = std::atoi(argv[i + 5]);
    p.n_vt = std::atoi(argv[i + 6]);
    p.cpu = std::atoi(argv[i + 7]);
    p.mc = std::atoi(argv[i + 8]);
    p.vc = std::atoi(argv[i + 9]);
    p.G2 = std::atoi(argv[i + 10]);
    p.spill_pct = std::atoi(argv[i + 11]);
    const int bm = bd::plan_bm(p, n_rows);
    const int n_mt = n_rows > 0 ? bd::cdiv(n_rows, bm) : 0;  // m-tiles
    const int n_rmt = bd::plan_runner_mts(p, n_rows);        // runner m-tiles (mc m-tiles each)
    int hdr[bd::HDR_WORDS] = {0};
    bd::plan_header(p, n_rows, hdr);  // what the compaction kernel stores
    const int slots = n_rows > 0 ? hdr[bd::HDR_SLOTS] : 0;
    const int vsplit = hdr[bd::HDR_VSPLIT];
    std::vector<int> cover(static_cast<size_t>(n_mt) * p.n_vt, 0);
    std::vector<int> slot_owner(static_cast<size_t>(slots > 0 ? slots : 1), -1);
    const char* fail = nullptr;
    if (hdr[bd::HDR_SLOTS] > bd::plan_max_slots(p)) fail = "more slots than the workspace holds";
    if (bd::plan_vc(p) == 2 && vsplit < p.n_vt && vsplit % 2 != 0) fail = "odd split with v-tile pairs";
    long long max_load[2] = {0, 0};
    for (int role = 0; role < 2 && !fail; ++role) {
      bd::BandPlan q = p;  // the launch's own arguments
      q.role = role;
      if (role == 1) {
        if (p.G2 <= 0 || vsplit == p.n_vt) break;  // no spill launch
        q.G = p.G2;
        q.mc = 1;
        q.vc = 1;
        q.cpu = bd::SPILL_UNIT_SLOTS;
      }
      const int mc = bd::plan_mc(q), vc = bd::plan_vc(q);
      const int unit_slots = bd::plan_unit_slots(q);
      const int gm = role ? hdr[bd::HDR_GM2] : hdr[bd::HDR_GM];
      const int gv = role ? hdr[bd::HDR_GV2] : hdr[bd::HDR_GV];
      const int lo = role ? vsplit : 0, hi = role ? p.n_vt : vsplit;
      const int runner_mts = bd::plan_runner_mts(q, n_rows);
      // the round of each (band, part): every unit of a part must run in the same round
      std::vector<int> part_round(static_cast<size_t>(bd::cdiv(runner_mts > 0 ? runner_mts : 1, gm > 0 ? gm : 1)) *
                                      (gv > 0 ? gv : 1), -1);
      for (int r = 0; r < q.G && !fail; ++r) {
        bd::TileIter it;
        it.init(q, hdr, r);
        long long load = 0;
        while (it.next_unit()) {
          if (it.m_tile < 0 || it.m_tile >= n_mt || it.m_tile % mc != 0) fail = "m-tile out of range";
          else if (it.part < 0 || it.part >= gv) fail = "part out of range";
          else if (it.vt >= it.vt_end) fail = "empty unit";
          if (fail) break;
          for (int sub = 0; sub < unit_slots && !fail; ++sub) {
            const int slot = it.slot0 + it.part * unit_slots + sub;
            if (slot < 0 || slot >= slots) fail = "slot beyond the partial slots";
            else if (slot_owner[slot] >= 0 && slot_owner[slot] != role) fail = "both launches write one slot";
            else slot_owner[slot] = role;
          }
          if (fail) break;
          int& pr = part_round[static_cast<size_t>(it.m_tile / mc / gm) * gv + it.part];
          if (pr >= 0 && pr != it.round) {
            fail = "the units of one part run in different rounds";
            break;
          }
          pr = it.round;
          for (int step = it.vt; step < it.vt_end && !fail; ++step)
            for (int s = 0; s < vc; ++s) {
              const int v = role ? step : step * vc + s;
              if (v < lo || v >= p.n_vt) {
                if (v < p.n_vt) fail = "v-tile outside the launch's range";
                continue;  // the discarded second v-tile of a step past the vocabulary
              }
              if (v >= hi) {
                fail = "v-tile outside the launch's range";
                break;
              }
              // the runner's mc m-tiles (one beyond the last is computed on no rows)
              for (int m = 0; m < mc && it.m_tile + m < n_mt; ++m) ++cover[static_cast<size_t>(it.m_tile + m) * p.n_vt + v];
            }
          load += it.vt_end - it.vt;
        }
        if (load > max_load[role]) max_load[role] = load;
      }
    }
    for (size_t k = 0; !fail && k < cover.size(); ++k)
      if (cover[k] != 1) fail = "a (m-tile, v-tile) pair is not taken exactly once";
    if (fail) {
      std::printf("FAIL %s\n", fail);
    } else {
      // the even share: time of a main runner's step = 1 (mc m-tiles x vc v-tiles on mc x vc pairs), of a
      // spill pair's v-tile = w
      const double w = (p.spill_pct > 0 ? p.spill_pct : 100) / 100.0;
      const double vcd = bd::plan_vc(p);
      const double ideal = p.G2 > 0 && n_rows > 0
                               ? w * n_mt * n_rmt * static_cast<double>(p.n_vt) / (p.G2 * n_rmt + w * n_mt * p.G * vcd)
                               : static_cast<double>(n_rmt) * p.n_vt / (p.G * vcd);
      std::printf("ok %d %d %d %lld %.3f %d %d %lld %d %d\n", n_mt, hdr[bd::HDR_GV], slots, max_load[0], ideal,
                  hdr[bd::HDR_GM], vsplit, max_load[1], hdr[bd::HDR_GM2], hdr[bd::HDR_GV2]);
    }
  }
  return 0;
}
