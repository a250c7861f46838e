// Host-side Task Scheduler of the FedOptima server (Algorithms 2 and 3) with
// the activation flow control of Sec. 3.4.1.
//
// State: one ring of batch-slot indices per device (Q^act_k), consumption
// counters c_k, Sender Status per device, a FIFO free list of the omega
// slots, and a FIFO of devices refused while their queue was empty.
//
// Readings where the paper is silent: argmin ties go to the lowest device
// index and only non-empty queues compete; both the global cap omega and a
// per-device ring depth are enforced; each dequeue also turns on the head
// of the blocked FIFO; a (re)joining device gets c_k = max(c_k, min over the
// other active devices).
#pragma once
#include <cstdint>
#include <vector>

namespace fo {

enum SchedPolicy { kCounter = 0, kFifo = 1 };

class TaskScheduler {
 public:
  // A depth above omega never binds (sum_k |Q_k| <= omega is reached
  // first), so the rings hold min(depth, omega) entries per device.
  TaskScheduler(int K, int omega, int depth, int policy)
      : K_(K), omega_(omega), depth_(depth < omega ? depth : omega), policy_(policy),
        ring_(size_t(K) * depth_), head_(K, 0), len_(K, 0), c_(K, 0),
        on_(K, 1), active_(K, 1), free_(omega), blocked_flag_(K, 0) {
    for (int i = 0; i < omega; ++i) free_[i] = i;
    free_head_ = 0;
    free_len_ = omega;
  }

  int K() const { return K_; }
  int omega() const { return omega_; }
  int queued_total() const { return total_; }
  int queued(int k) const { return len_[k]; }
  const std::vector<uint64_t>& counters() const { return c_; }
  const std::vector<uint8_t>& sender_on() const { return on_; }
  bool active(int k) const { return active_[k] != 0; }

  // What put(k) would do, without changing any state: 0 = it would accept
  // (slot set to the slot it would hand out), 2 = it would refuse, -1 = bad
  // argument.  Lets a caller fill the slot before committing the upload.
  int peek(int k, int32_t* slot) const {
    if (k < 0 || k >= K_ || !active_[k]) return -1;
    if (total_ >= omega_ || len_[k] >= depth_) return 2;
    *slot = free_[free_head_];
    return 0;
  }

  // put(): returns 0 = accepted (slot set), 2 = refused (cap/depth), -1 bad arg.
  int put(int k, int32_t* slot) {
    if (k < 0 || k >= K_ || !active_[k]) return -1;
    if (total_ >= omega_ || len_[k] >= depth_) {
      on_[k] = 0;
      if (len_[k] == 0 && !blocked_flag_[k]) {
        blocked_.push_back(k);
        blocked_flag_[k] = 1;
      }
      return 2;
    }
    int32_t s = free_[free_head_];
    free_head_ = (free_head_ + 1) % omega_;
    --free_len_;
    ring_[size_t(k) * depth_ + (head_[k] + len_[k]) % depth_] = s;
    ++len_[k];
    ++total_;
    if (policy_ == kFifo) arrivals_.push_back(k);
    if (blocked_flag_[k]) remove_blocked(k);
    on_[k] = (total_ < omega_ && len_[k] < depth_) ? 1 : 0;
    *slot = s;
    return 0;
  }

  // get(): returns 0 = served (k, slot set), 1 = every queue empty.
  int get(int* k_out, int32_t* slot) {
    int k = -1;
    if (policy_ == kCounter) {
      for (int j = 0; j < K_; ++j)
        if (len_[j] > 0 && (k < 0 || c_[j] < c_[k])) k = j;
    } else if (arr_head_ < arrivals_.size()) {
      k = arrivals_[arr_head_++];
      if (arr_head_ > 4096 && arr_head_ * 2 > arrivals_.size()) {
        arrivals_.erase(arrivals_.begin(), arrivals_.begin() + arr_head_);
        arr_head_ = 0;
      }
    }
    if (k < 0) return 1;
    int32_t s = ring_[size_t(k) * depth_ + head_[k]];
    head_[k] = (head_[k] + 1) % depth_;
    --len_[k];
    --total_;
    ++c_[k];
    free_[(free_head_ + free_len_) % omega_] = s;
    ++free_len_;
    on_[k] = 1;
    if (blocked_head_ < blocked_.size()) {
      int j = blocked_[blocked_head_++];
      blocked_flag_[j] = 0;
      on_[j] = 1;
      compact_blocked();
    }
    *k_out = k;
    *slot = s;
    return 0;
  }

  int set_active(int k, int active) {
    if (k < 0 || k >= K_) return -1;
    if (active && !active_[k]) {
      bool any = false;
      uint64_t lo = 0;
      for (int j = 0; j < K_; ++j) {
        if (j == k || !active_[j]) continue;
        if (!any || c_[j] < lo) lo = c_[j];
        any = true;
      }
      if (any && c_[k] < lo) c_[k] = lo;
      active_[k] = 1;
      on_[k] = 1;
    } else if (!active && active_[k]) {
      active_[k] = 0;
      on_[k] = 0;
      if (blocked_flag_[k]) remove_blocked(k);
    }
    return 0;
  }

 private:
  void remove_blocked(int k) {
    for (size_t i = blocked_head_; i < blocked_.size(); ++i)
      if (blocked_[i] == k) {
        blocked_.erase(blocked_.begin() + i);
        break;
      }
    blocked_flag_[k] = 0;
  }
  void compact_blocked() {
    if (blocked_head_ > 64 && blocked_head_ * 2 > blocked_.size()) {
      blocked_.erase(blocked_.begin(), blocked_.begin() + blocked_head_);
      blocked_head_ = 0;
    }
  }

  int K_, omega_, depth_, policy_;
  std::vector<int32_t> ring_;
  std::vector<int> head_, len_;
  std::vector<uint64_t> c_;
  std::vector<uint8_t> on_, active_;
  std::vector<int32_t> free_;
  int free_head_ = 0, free_len_ = 0, total_ = 0;
  std::vector<int> blocked_;
  size_t blocked_head_ = 0;
  std::vector<uint8_t> blocked_flag_;
  std::vector<int> arrivals_;
  size_t arr_head_ = 0;
};

}  // namespace fo
