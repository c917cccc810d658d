// Host check of the LM-head work plan (common.cuh): for each case given on
// the command line as "n_rows BM GM vt_kb row_bytes G n_vt cpu mc", every (m-tile,
// v-tile) pair is taken by exactly one unit, the units of every part run in
// the same round, the part indices stay below the partial slots the merge
// reads, and the busiest runner's v-tiles are reported against the even
// share. Prints one line per case:
//   ok <n_mt> <gv> <slots> <max_vtiles> <ideal_vtiles>   or   FAIL <reason>
#include <cstdio>
#include <cstdlib>
#include <vector>

#include "common.cuh"

int main(int argc, char** argv) {
  for (int i = 1; i + 8 < argc; i += 9) {
    bd::BandPlan p;
    const int n_rows = std::atoi(argv[i]);
    p.BM = std::atoi(argv[i + 1]);
    p.GM = std::atoi(argv[i + 2]);
    p.vt_kb = std::atoi(argv[i + 3]);
    p.row_bytes = std::atoi(argv[i + 4]);
    p.G = std::atoi(argv[i + 5]);
    p.n_vt = std::atoi(argv[i + 6]);
    p.cpu = std::atoi(argv[i + 7]);
    p.mc = std::atoi(argv[i + 8]);
    p.gv_fixed = 0;
    p.rr = 0;
    const int bm = bd::plan_bm(p, n_rows);
    const int n_mt = n_rows > 0 ? bd::cdiv(n_rows, bm) : 0;  // m-tiles
    const int n_rmt = bd::plan_runner_mts(p, n_rows);        // runner m-tiles (mc m-tiles each)
    const int mc = bd::plan_mc(p);
    std::vector<int> cover(static_cast<size_t>(n_mt) * p.n_vt, 0);
    int gm = 1, gv = 1;
    bd::plan_choose(p, n_rows, &gm, &gv);  // what the compaction kernel stores beside N
    const int slots = n_rows > 0 ? gv * p.cpu : 0;
    // the round of each (band, part): every unit of a part must run in the same round
    std::vector<int> part_round(static_cast<size_t>(bd::cdiv(n_rmt > 0 ? n_rmt : 1, gm)) * gv, -1);
    const char* fail = nullptr;
    long long max_load = 0;
    for (int r = 0; r < p.G && !fail; ++r) {
      bd::TileIter it;
      it.init(p, n_rows, gm, gv, r);
      long long load = 0;
      while (it.next_unit()) {
        if (it.m_tile < 0 || it.m_tile >= n_mt || it.m_tile % mc != 0) fail = "m-tile out of range";
        else if ((it.part + 1) * p.cpu > slots) fail = "part beyond the partial slots";
        else if (it.vt < 0 || it.vt_end > p.n_vt || it.vt >= it.vt_end) fail = "empty or out-of-range v-tiles";
        if (fail) break;
        int& pr = part_round[static_cast<size_t>(it.m_tile / mc / gm) * gv + it.part];
        if (pr >= 0 && pr != it.round) {
          fail = "the units of one part run in different rounds";
          break;
        }
        pr = it.round;
        // the runner's mc m-tiles (one beyond the last is computed on no rows)
        for (int q = 0; q < mc && it.m_tile + q < n_mt; ++q)
          for (int v = it.vt; v < it.vt_end; ++v) ++cover[static_cast<size_t>(it.m_tile + q) * p.n_vt + v];
        load += it.vt_end - it.vt;
      }
      if (load > max_load) max_load = load;
    }
    for (size_t k = 0; !fail && k < cover.size(); ++k)
      if (cover[k] != 1) fail = "a (m-tile, v-tile) pair is not taken exactly once";
    if (fail) {
      std::printf("FAIL %s\n", fail);
    } else {
      std::printf("ok %d %d %d %lld %.3f %d\n", n_mt, slots / (p.cpu > 0 ? p.cpu : 1), slots, max_load,
                  static_cast<double>(n_rmt) * p.n_vt / p.G, gm);
    }
  }
  return 0;
}
