// Committed length of an append-only KV cache under asynchronous appends (Sec. 3.3:
// the fast system ticks on the cache as it stands while the slow system appends the
// newest frame's tokens behind it). Host-only bookkeeping, no CUDA: appends are
// reserved in order, each owns rows [first, first + n), they complete in the order
// they were issued (one stream), and a tick may read exactly the rows of completed
// appends -- its snapshot. Rows being written always lie at or past the snapshot, so
// the cache needs no lock.
#pragma once

#include <deque>

namespace fsx {

template <typename Token>
class SnapshotLedger {
 public:
  SnapshotLedger(long long committed, long long capacity) : committed_(committed), end_(committed), capacity_(capacity) {}

  // Rows for the next append of n rows: its first row, or -1 when they would pass the
  // capacity (nothing is reserved then).
  long long reserve(long long n, Token token) {
    if (n <= 0 || end_ + n > capacity_) return -1;
    const long long first = end_;
    end_ += n;
    pending_.push_back(Pending{end_, token});
    return first;
  }

  // Retire completed appends in issue order; done(token) tells whether one has completed.
  // Returns the committed length afterwards.
  template <typename DoneFn>
  long long poll(DoneFn done) {
    while (!pending_.empty() && done(pending_.front().token)) {
      committed_ = pending_.front().end;
      pending_.pop_front();
    }
    return committed_;
  }

  long long committed() const { return committed_; }  // rows a tick may read
  long long end() const { return end_; }              // committed + rows of appends in flight
  int in_flight() const { return static_cast<int>(pending_.size()); }
  bool empty() const { return pending_.empty(); }
  Token oldest() const { return pending_.front().token; }

 private:
  struct Pending {
    long long end;
    Token token;
  };
  long long committed_, end_, capacity_;
  std::deque<Pending> pending_;
};

}  // namespace fsx
