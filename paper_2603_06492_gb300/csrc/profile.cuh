// Optional per-kernel-class timing with CUDA events, recorded on the stream
// each kernel is launched on.  Off by default; when on, every launch made by
// the library is bracketed by two events and attributed to a class with its
// algorithmic FLOPs and bytes, so a caller can compute achieved throughput of
// each kernel live, inside its own timed region.
#pragma once

#include <cuda_runtime.h>

#include <map>
#include <mutex>
#include <string>
#include <vector>

namespace noble {

enum Bound : int { kBoundTensor = 0, kBoundHbm = 1, kBoundAlu = 2 };

struct KernelInfo {
    const char *name;  // kernel class
    int bound;         // Bound
    double flops;      // algorithmic FLOPs of this launch
    double bytes;      // algorithmic DRAM bytes of this launch
};

class Profiler {
  public:
    static Profiler &get()
    {
        static Profiler p;
        return p;
    }
    void enable(bool on) { std::lock_guard<std::mutex> g(mu_); on_ = on; }
    bool on() const { return on_; }
    void reset()
    {
        std::lock_guard<std::mutex> g(mu_);
        collect_locked();
        agg_.clear();
    }
    // Returns a pending slot (or -1 when off); record the begin event.
    int begin(cudaStream_t st)
    {
        if (!on_) return -1;
        std::lock_guard<std::mutex> g(mu_);
        int slot;
        if (!free_.empty()) {
            slot = free_.back();
            free_.pop_back();
        } else {
            Pair p{};
            if (cudaEventCreate(&p.a) != cudaSuccess || cudaEventCreate(&p.b) != cudaSuccess) {
                cudaGetLastError();
                return -1;
            }
            pairs_.push_back(p);
            slot = (int)pairs_.size() - 1;
        }
        cudaEventRecord(pairs_[slot].a, st);
        return slot;
    }
    void end(int slot, cudaStream_t st, const KernelInfo &ki)
    {
        if (slot < 0) return;
        std::lock_guard<std::mutex> g(mu_);
        cudaEventRecord(pairs_[slot].b, st);
        pending_.push_back({slot, ki});
    }
    struct Entry {
        std::string name;
        int bound = 0;
        uint64_t launches = 0;
        double ms = 0, flops = 0, bytes = 0;
    };
    std::vector<Entry> read()
    {
        std::lock_guard<std::mutex> g(mu_);
        collect_locked();
        std::vector<Entry> out;
        for (auto &kv : agg_) out.push_back(kv.second);
        return out;
    }

  private:
    struct Pair {
        cudaEvent_t a, b;
    };
    struct Pending {
        int slot;
        KernelInfo ki;
    };
    void collect_locked()
    {
        for (auto &p : pending_) {
            cudaEventSynchronize(pairs_[p.slot].b);
            float ms = 0;
            cudaEventElapsedTime(&ms, pairs_[p.slot].a, pairs_[p.slot].b);
            Entry &e = agg_[p.ki.name];
            e.name = p.ki.name;
            e.bound = p.ki.bound;
            e.launches += 1;
            e.ms += ms;
            e.flops += p.ki.flops;
            e.bytes += p.ki.bytes;
            free_.push_back(p.slot);
        }
        pending_.clear();
        cudaGetLastError();
    }
    std::mutex mu_;
    bool on_ = false;
    std::vector<Pair> pairs_;
    std::vector<int> free_;
    std::vector<Pending> pending_;
    std::map<std::string, Entry> agg_;
};

}  // namespace noble
