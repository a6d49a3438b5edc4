// Randomised schedules of appends, completions and ticks against SnapshotLedger (the
// committed-length bookkeeping of the asynchronous fast-slow session). Every tick's
// snapshot must cover exactly the rows of completed appends, no row of an append in
// flight may lie inside a snapshot, reserved ranges must be contiguous and disjoint,
// and nothing may be reserved past the capacity. Prints "ok <ticks>" or the failure.
#include <cstdio>
#include <cstdlib>
#include <random>
#include <set>
#include <vector>

#include "ledger.h"

int main(int argc, char** argv) {
  const int seeds = argc > 1 ? std::atoi(argv[1]) : 200;
  long long ticks = 0;
  for (int seed = 0; seed < seeds; ++seed) {
    std::mt19937 rng(seed);
    const long long committed0 = rng() % 300;
    const long long capacity = committed0 + 4 * (rng() % 40);
    fsx::SnapshotLedger<int> ledger(committed0, capacity);
    std::set<int> done;                       // completed append tokens
    struct Range { long long first, end; int token; };
    std::vector<Range> ranges;                // every reserved append, in issue order
    int next_token = 0, next_complete = 0;    // appends complete in issue order
    long long last_snapshot = committed0, expect_end = committed0;
    for (int step = 0; step < 400; ++step) {
      const int op = rng() % 3;
      if (op == 0) {                          // an append of 4 rows (every K ticks in the paper)
        const int tok = next_token;
        const long long first = ledger.reserve(4, tok);
        if (expect_end + 4 > capacity) {
          if (first != -1) { std::printf("seed %d: reserved past the capacity\n", seed); return 1; }
          continue;
        }
        if (first != expect_end) { std::printf("seed %d: non-contiguous reservation\n", seed); return 1; }
        ranges.push_back({first, first + 4, tok});
        expect_end += 4;
        ++next_token;
      } else if (op == 1) {                   // the oldest append in flight completes
        if (next_complete < next_token) done.insert(next_complete++);
      } else {                                // a tick takes its snapshot
        const long long snap = ledger.poll([&](int t) { return done.count(t) > 0; });
        ++ticks;
        long long expect = committed0;
        for (const Range& r : ranges)
          if (done.count(r.token)) expect = r.end;
        if (snap != expect) { std::printf("seed %d: snapshot %lld, completed rows end at %lld\n", seed, snap, expect); return 1; }
        for (const Range& r : ranges)
          if (!done.count(r.token) && r.first < snap) {
            std::printf("seed %d: snapshot %lld includes rows of an append in flight\n", seed, snap);
            return 1;
          }
        if (snap < last_snapshot) { std::printf("seed %d: snapshot went backwards\n", seed); return 1; }
        last_snapshot = snap;
        if (ledger.end() != expect_end || ledger.in_flight() != next_token - (int)done.size()) {
          std::printf("seed %d: reserved end or in-flight count wrong\n", seed);
          return 1;
        }
      }
    }
  }
  std::printf("ok %lld\n", ticks);
  return 0;
}
