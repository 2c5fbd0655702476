// A round's host-side state in one call and one buffer: the GP state
// (Section 4.3), the packed forest (Eq. 3) and, for EHVI, the box
// decomposition of the region the front does not dominate (Section 4.4)
// with the base samples, or the boxes' grid index for the exact EHVI.  The
// fp64 GP factorisation (objectives in parallel) and the forest's packing run
// on the library's host threads while the calling thread decomposes the
// boxes, so the round's host time is the longest of them rather than their
// sum.
#include <algorithm>
#include <atomic>
#include <chrono>
#include <condition_variable>
#include <cstring>
#include <deque>
#include <functional>
#include <mutex>
#include <thread>
#include <vector>

#include <unistd.h>

#include "internal.h"

namespace {

constexpr int64_t kSlotAlign = 256;

int64_t slot(int64_t bytes) { return (bytes + kSlotAlign - 1) / kSlotAlign * kSlotAlign; }

// A few background threads shared by the library's host preparation.  A
// job is a function; parallel_for runs f(0 .. count-1) over the pool and the
// calling thread, and a caller that waits runs queued jobs meanwhile, so
// nested use (a job that itself calls parallel_for) cannot deadlock.
class Pool {
public:
    // A process forked after the threads started has none of them: it makes
    // its own pool (the old object is left alone).
    static Pool& get() {
        static std::mutex make_mu;
        static Pool* p = nullptr;
        static pid_t owner = 0;
        std::lock_guard<std::mutex> lk(make_mu);
        if (!p || owner != getpid()) {
            p = new Pool();  // never destroyed: no join at static destruction time
            owner = getpid();
        }
        return *p;
    }

    struct Latch {
        std::atomic<int> left{0};
    };

    void submit(std::function<void()> job, Latch* latch) {
        latch->left.fetch_add(1);
        bool wake;
        {
            std::lock_guard<std::mutex> lk(mu_);
            jobs_.push_back({std::move(job), latch});
            pending_.fetch_add(1);
            wake = sleepers_ > 0;
        }
        if (wake) cv_.notify_one();
    }

    // Until latch reaches zero: run queued jobs, else sleep briefly.
    void wait(Latch* latch) {
        while (latch->left.load() > 0) {
            if (!run_one()) {
                std::unique_lock<std::mutex> lk(mu_);
                done_cv_.wait_for(lk, std::chrono::microseconds(50), [&] { return latch->left.load() == 0; });
            }
        }
    }

    int threads() const { return n_threads_; }

private:
    struct Job {
        std::function<void()> fn;
        Latch* latch;
    };

    Pool() {
        const unsigned hw = std::thread::hardware_concurrency();
        n_threads_ = hw > 1 ? (int)std::min(hw - 1, 7u) : 1;
        for (int t = 0; t < n_threads_; ++t) std::thread([this] { loop(); }).detach();
    }

    bool run_one() {
        Job job;
        {
            std::lock_guard<std::mutex> lk(mu_);
            if (jobs_.empty()) return false;
            job = std::move(jobs_.front());
            jobs_.pop_front();
            pending_.fetch_sub(1);
        }
        job.fn();
        if (job.latch->left.fetch_sub(1) == 1) {
            std::lock_guard<std::mutex> lk(mu_);
            done_cv_.notify_all();
        }
        return true;
    }

    // After each job a thread polls for the next one for kSpin before it
    // sleeps: waking a sleeping thread takes tens of microseconds, as long as
    // the jobs themselves.
    void loop() {
        for (;;) {
            const auto until = std::chrono::steady_clock::now() + kSpin;
            while (pending_.load() == 0 && std::chrono::steady_clock::now() < until) std::this_thread::yield();
            if (pending_.load() == 0) {
                std::unique_lock<std::mutex> lk(mu_);
                ++sleepers_;
                cv_.wait(lk, [&] { return !jobs_.empty(); });
                --sleepers_;
            }
            run_one();
        }
    }

    static constexpr std::chrono::microseconds kSpin{500};

    std::mutex mu_;
    std::condition_variable cv_, done_cv_;
    std::deque<Job> jobs_;
    std::atomic<int> pending_{0};  // jobs queued, readable without the lock
    int sleepers_ = 0;             // threads waiting on cv_ (under mu_)
    int n_threads_ = 1;
};

}  // namespace

void scoot_host_parallel(int count, const std::function<void(int)>& fn) {
    if (count <= 0) return;
    if (count == 1) {
        fn(0);
        return;
    }
    Pool& pool = Pool::get();
    Pool::Latch latch;
    for (int i = 1; i < count; ++i) pool.submit([&fn, i] { fn(i); }, &latch);
    fn(0);
    pool.wait(&latch);
}

extern "C" {

scoot_status scoot_round_state_build(const scoot_round_inputs* in, void* h_buf, int64_t cap, scoot_round_state* out) {
    if (!in || !out || (cap > 0 && !h_buf) || cap < 0) return SCOOT_EINVAL;
    std::memset(out, 0, sizeof(*out));
    out->off_gp = out->off_forest = out->off_box_lo = out->off_box_hi = out->off_eps = -1;
    out->off_grid = out->off_corner = out->off_fant = -1;
    if (!in->space || !in->x_obs || !in->y || !in->nodes || !in->tree_offset) return SCOOT_EINVAL;
    if (in->boxes < 0 || in->boxes > 2) return SCOOT_EINVAL;
    const int M = in->n_obj, n = in->n;
    scoot_status s = scoot_gp_layout_init(in->space, n, in->d, M, in->kernel, &out->gp);
    if (s != SCOOT_OK) return s;
    s = scoot_forest_layout_init(in->nodes, in->tree_offset, in->n_trees, in->d, in->leaf_scale, &out->forest);
    if (s != SCOOT_OK) return s;
    int64_t off = 0;
    if (!in->gp_on_device) {
        out->off_gp = off;
        off += slot(out->gp.bytes);
    }
    char* buf = static_cast<char*>(h_buf);
    // The fantasy state: its header and front now, its fp64 arrays from the
    // GP job's own factorisation.
    void* fant = nullptr;
    if (in->fantasy_q > 0) {
        if (in->gp_on_device || in->warp || !in->ref) return SCOOT_EINVAL;
        FantHeader fl;
        scoot_fant_layout(n, in->d, M, in->fantasy_q, &fl);
        out->off_fant = off;
        off += slot(fl.bytes);
        if (out->off_fant + fl.bytes <= cap) {
            s = scoot_fant_header(in->space, &out->gp, in->y, in->signal_var, in->noise_var, in->ref, in->fantasy_q,
                                  buf + out->off_fant, fl.bytes);
            if (s != SCOOT_OK) return s;
            fant = buf + out->off_fant;
            out->fant_box_cap = static_cast<const FantHeader*>(fant)->box_cap;
        }
    }
    // The GP factorisation first, on the worker, if its slot fits.
    scoot_status gp_status = SCOOT_OK;
    Pool::Latch latch;
    const bool gp_job = !in->gp_on_device && out->gp.bytes <= cap;
    if (gp_job) {
        double* cond = out->cond;
        const scoot_round_inputs* pin = in;
        const scoot_gp_layout* gl = &out->gp;
        Pool::get().submit([pin, gl, buf, cond, fant, &gp_status] {
            gp_status = scoot_gp_build(pin->space, pin->x_obs, pin->ld_obs, pin->y, pin->lengthscale,
                                       pin->signal_var, pin->noise_var, pin->warp, gl, buf, cond, fant);
        }, &latch);
    }
    auto finish = [&](scoot_status st) {
        if (gp_job) Pool::get().wait(&latch);
        if (st == SCOOT_OK && gp_status != SCOOT_OK) st = gp_status;
        return st;
    };
    out->off_forest = off;
    off += slot(out->forest.bytes);
    // The forest's packing on another thread while this one builds the boxes.
    scoot_status forest_status = SCOOT_OK;
    Pool::Latch forest_latch;
    const bool forest_job = out->off_forest + out->forest.bytes <= cap;
    if (forest_job) {
        const scoot_round_inputs* pin = in;
        const scoot_forest_layout* fl = &out->forest;
        char* dst = buf + out->off_forest;
        Pool::get().submit([pin, fl, dst, &forest_status] {
            forest_status = scoot_forest_pack(fl, pin->nodes, pin->tree_offset, dst);
        }, &forest_latch);
    }
    auto finish_all = [&](scoot_status st) {
        if (forest_job) Pool::get().wait(&forest_latch);
        if (st == SCOOT_OK && forest_status != SCOOT_OK) st = forest_status;
        return finish(st);
    };
    std::vector<float> lo, hi, grid;
    std::vector<uint32_t> corner;
    if (in->boxes) {
        if (M < 2 || !in->ref) return finish_all(SCOOT_EINVAL);
        int32_t nb = 0, fs = 0, bcap = 1024;
        for (;;) {
            lo.assign((size_t)bcap * M, 0.0f);
            hi.assign((size_t)bcap * M, 0.0f);
            s = scoot_boxes_build(in->y, n, M, in->ref, bcap, lo.data(), hi.data(), &nb, &fs);
            if (s == SCOOT_EUNSUPPORTED && nb > bcap) {  // capacity: nb holds the count needed
                bcap = nb;
                continue;
            }
            if (s != SCOOT_OK) return finish_all(s);
            break;
        }
        out->n_boxes = nb;
        out->front_size = fs;
        out->off_box_lo = off;
        off += slot((int64_t)nb * M * 4);
        out->off_box_hi = off;
        off += slot((int64_t)nb * M * 4);
        if (in->boxes == 1) {
            if (!in->eps || in->n_mc < 1) return finish_all(SCOOT_EINVAL);
            out->off_eps = off;
            off += slot((int64_t)in->n_mc * M * 4);
        } else {
            const int gc = in->grid_cap > 0 ? in->grid_cap : 256;
            grid.assign((size_t)M * gc, 0.0f);
            corner.assign((size_t)(nb > 0 ? nb : 1) * M, 0u);
            s = scoot_boxes_index(lo.data(), hi.data(), nb, M, gc, grid.data(), out->n_grid, corner.data());
            if (s != SCOOT_OK) return finish_all(s);
            out->grid_cap = gc;
            out->off_grid = off;
            off += slot((int64_t)M * gc * 4);
            out->off_corner = off;
            off += slot((int64_t)nb * M * 4);
        }
    }
    out->bytes = off;
    if (off > cap) return finish_all(SCOOT_ENOMEM);  // out->bytes holds the size needed
    if (in->boxes) {
        std::memcpy(buf + out->off_box_lo, lo.data(), (size_t)out->n_boxes * M * 4);
        std::memcpy(buf + out->off_box_hi, hi.data(), (size_t)out->n_boxes * M * 4);
        if (in->boxes == 1) {
            std::memcpy(buf + out->off_eps, in->eps, (size_t)in->n_mc * M * 4);
        } else {
            std::memcpy(buf + out->off_grid, grid.data(), grid.size() * 4);
            std::memcpy(buf + out->off_corner, corner.data(), (size_t)out->n_boxes * M * 4);
        }
    }
    return finish_all(s);
}

}  // extern "C"
