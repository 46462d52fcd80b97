/*
 * Thread pool for the host side of staging (copies of pageable sources and callback fills into
 * pinned slots).  Host-only C++; no CUDA.
 */
#ifndef CFA_POOL_H
#define CFA_POOL_H

#include <atomic>
#include <condition_variable>
#include <cstdint>
#include <functional>
#include <mutex>
#include <thread>
#include <vector>

namespace cfa {

/*
 * run(n, f) executes f(0) .. f(n-1) on the pool's threads and the calling thread.  Each run owns
 * a Job on the caller's stack; a worker joins a job only while it is published, under the
 * mutex, and run() returns only when every part is done and every worker has left the job, so
 * no worker can touch a finished job or take a part of the next one with a stale counter.
 */
class Pool {
  public:
    explicit Pool(int n)
    {
        for (int i = 0; i < n; ++i) threads_.emplace_back([this] { loop(); });
    }
    ~Pool()
    {
        {
            std::lock_guard<std::mutex> g(mu_);
            stop_ = true;
        }
        cv_.notify_all();
        for (auto &t : threads_) t.join();
    }
    void run(int nparts, const std::function<void(int)> &f)
    {
        if (threads_.empty() || nparts <= 1) {
            for (int k = 0; k < nparts; ++k) f(k);
            return;
        }
        Job job(&f, nparts);
        {
            std::lock_guard<std::mutex> g(mu_);
            job_ = &job;
            ++gen_;
        }
        cv_.notify_all();
        work(&job);
        std::unique_lock<std::mutex> lk(mu_);
        done_.wait(lk, [&] { return job.pending.load() == 0 && job.users == 0; });
        job_ = nullptr;
    }

  private:
    struct Job {
        Job(const std::function<void(int)> *f, int n) : fn(f), total(n), pending(n) {}
        const std::function<void(int)> *fn;
        const int total;
        std::atomic<int> next{0};
        std::atomic<int> pending;
        int users = 0; /* workers inside the job; guarded by mu_ */
    };
    void work(Job *j)
    {
        for (;;) {
            const int k = j->next.fetch_add(1);
            if (k >= j->total) return;
            (*j->fn)(k);
            if (j->pending.fetch_sub(1) == 1) {
                std::lock_guard<std::mutex> g(mu_);
                done_.notify_all();
            }
        }
    }
    void loop()
    {
        uint64_t seen = 0;
        for (;;) {
            Job *j;
            {
                std::unique_lock<std::mutex> lk(mu_);
                cv_.wait(lk, [&] { return stop_ || gen_ != seen; });
                if (stop_) return;
                seen = gen_;
                j = job_;
                if (!j) continue;
                ++j->users;
            }
            work(j);
            {
                std::lock_guard<std::mutex> g(mu_);
                --j->users;
            }
            done_.notify_all();
        }
    }
    std::vector<std::thread> threads_;
    std::mutex mu_;
    std::condition_variable cv_, done_;
    Job *job_ = nullptr;
    uint64_t gen_ = 0;
    bool stop_ = false;
};

} // namespace cfa

#endif /* CFA_POOL_H */
