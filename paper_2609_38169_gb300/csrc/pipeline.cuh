// The persistent page pipeline shared by the fused decode kernels.
//
// Each CTA walks the items first, first + G, first + 2G, ... of one launch
// (item = head * nb + batch entry, head-major so that concurrently resident
// CTAs mostly work on one head). The last warp keeps up to S-1 items in
// flight: their copies land in a ring of S shared-memory stages and complete on
// one mbarrier per stage. The page travels as one bulk copy; the small vectors
// go as cp.async copies of 16 bytes per lane, which the whole warp issues at
// once. Every thread consumes the current stage, the page is rewritten in
// place, and lane 0 of the last warp (the producer thread) writes it back with
// a bulk store.
//
// Every wait is bounded: a stage whose copies do not land within the launch's
// limit (Shape::wait_cycles, kWaitCycles unless a test lowers it) raises
// STEPQ_ERR_TIMEOUT (the CTA agrees on it at its first barrier of the item),
// and the producer then waits, again with the bound, for this CTA's copies
// still in flight before the CTA returns. Should one of those waits give up as
// well, the CTA returns with that stage's copies possibly still in flight: the
// launch's results are then undefined, which the error status reports.
#pragma once

#include <cstdint>

#include "async.cuh"
#include "device.cuh"

namespace stepq {
namespace pipe {

constexpr long long kWaitCycles = 2000000000LL;      // ~1 s at 2 GHz
constexpr int kProducer = kThreads - 32;              // lane 0 of the last warp: page copies, stores
constexpr int kMaxStages = 4;                         // bars[0..4) barriers, bars[4..8) slot ids

// Repeated slot ids (two entries of one call writing one page race): every
// unordered pair of batch entries is compared once across the whole grid --
// entry i against entries i+1 .. i+floor(nb/2), cyclically -- and a repeated
// valid id raises STEPQ_ERR_DUP_SLOT. The check keeps no state, so launches that
// overlap on other streams or replay in a graph cannot disturb it. It costs about
// nb^2 / 2 comparisons per launch, a few per thread for nb = 1024.
__device__ __forceinline__ void check_repeats(const int32_t *slots, int nb, int pool_slots,
                                              unsigned int *err) {
    const long long half = nb / 2, pairs = (long long)nb * half;
    const long long threads = (long long)gridDim.x * blockDim.x;
    const long long chunk = (pairs + threads - 1) / threads;
    long long p = ((long long)blockIdx.x * blockDim.x + threadIdx.x) * chunk;
    const long long end = p + chunk < pairs ? p + chunk : pairs;
    if (p >= end) return;
    int i = (int)(p / half), d = (int)(p - (long long)i * half) + 1;
    int si = slots[i];
    for (; p < end; p++) {
        const int j = i + d < nb ? i + d : i + d - nb;
        if (slots[j] == si && si >= 0 && si < pool_slots) {
            raise_error(err, STEPQ_ERR_DUP_SLOT);
            return;
        }
        if (++d > half) {
            d = 1;
            si = slots[++i < nb ? i : 0];
        }
    }
}

// (head, batch entry) of item = head * nb + entry, stepped by the grid stride
// G = gq * nb + gr without divisions.
struct Cursor {
    int item, h, b;
    __device__ __forceinline__ Cursor(int it, int nb) : item(it), h(it / nb), b(it - (it / nb) * nb) {}
    __device__ __forceinline__ void step(int G, int gq, int gr, int nb) {
        item += G;
        h += gq;
        b += gr;
        if (b >= nb) {
            b -= nb;
            h++;
        }
    }
};

struct Shape {
    int items, nb, n_stages;
    const int32_t *slots;
    int pool_slots;
    unsigned int *err;
    long long wait_cycles;   // bound of every wait
    int withhold;            // test switch: the item whose copies never start, or -1
};

// Runs the item loop of this CTA (all threads call it; bars[0..S) initialised,
// S <= kMaxStages; the 16 bytes at bars + kMaxStages are free for the slot id of
// each stage, which the producer writes when it starts the stage and every
// thread reads once the stage's barrier has completed).
//   issue(h, b, slot, s, lane) all 32 lanes of the last warp: start the item's
//                             copies into stage s. Every lane's cp.async copies
//                             join the phase of bars[s] (cp_async_mbar_arrive)
//                             before the warp synchronises; lane 0 then arrives
//                             with expect_tx and starts the bulk copy of the page
//   process(h, b, slot, s, ok, refill) -> bool
//                             all threads: the step on stage s; must call
//                             refill() once, and return false from its first
//                             CTA barrier (which takes the OR of !ok) if a copy
//                             stalled
//   store(h, slot, s)         producer thread only: write the final page back
// An item whose slot id is out of range raises STEPQ_ERR_SLOT_RANGE; its stage
// completes without data and nothing is written. A slot id repeated within the
// launch raises STEPQ_ERR_DUP_SLOT (check_repeats); the pages of that slot are
// then undefined.
template <class Issue, class Process, class Store>
__device__ __forceinline__ void run(const Shape &p, uint64_t *bars, Issue &&issue, Process &&process,
                                    Store &&store) {
    const int tid = threadIdx.x;
    const int G = gridDim.x, S_n = p.n_stages;
    const int gq = G / p.nb, gr = G - gq * p.nb;
    const int first = blockIdx.x;
    const auto slot_ok = [&](int slot) { return slot >= 0 && slot < p.pool_slots; };
    volatile int *stage_slot = (volatile int *)(bars + kMaxStages);
    const int lane = tid & 31;
    const bool producer_warp = tid >= kProducer;
    const auto start = [&](int h, int b, int slot, int s) {
        if (lane == 0) stage_slot[s] = slot;
        if (h * p.nb + b == p.withhold) {
            // test switch: the stage expects bytes that never come, so its wait runs out
            if (lane == 0) mbar_arrive_tx(&bars[s], 16);
        } else if (slot_ok(slot)) {
            issue(h, b, slot, s, lane);
        } else if (lane == 0) {
            mbar_arrive(&bars[s]);
        }
    };
    // With three or more stages a stage is refilled two items after its own item
    // (its store has long finished reading it); with two stages, one item after.
    const int lag = S_n >= 3 ? 2 : 1;
    if (producer_warp) {
        Cursor c0(first, p.nb);
        for (int s = 0; s < S_n && c0.item < p.items; s++) {
            start(c0.h, c0.b, p.slots[c0.b], s);
            c0.step(G, gq, gr, p.nb);
        }
    }
    check_repeats(p.slots, p.nb, p.pool_slots, p.err);
    __syncthreads();                      // the first stages' slot ids are visible to every thread
    // iteration n >= lag refills stage (n - lag) mod S with item n - lag + S
    Cursor cur(first, p.nb), iss(first + S_n * G, p.nb);
    int s = 0, is = 0;                    // stage of the current item, stage refilled next
    uint32_t parity = 0;
    for (int n = 0; cur.item < p.items; n++) {
        Cursor nxt = cur;
        nxt.step(G, gq, gr, p.nb);
        // prefetch: the slot of the item this iteration will issue (producer)
        const bool do_issue = n >= lag && iss.item < p.items;
        int islot = -1;
        if (producer_warp && do_issue) islot = p.slots[iss.b];

        const bool ok = mbar_wait(&bars[s], parity, p.wait_cycles);
        // the item's slot id: the producer wrote it when it started the stage,
        // before at least one CTA barrier
        const int slot = stage_slot[s];
        const bool valid = slot_ok(slot);
        if (!valid && tid == 0) raise_error(p.err, STEPQ_ERR_SLOT_RANGE);
        // Refill the stage of an earlier item (its store was committed `lag`
        // items ago) with the item S-1 ahead of it: S-1 items stay in flight.
        const auto refill = [&start, tid, producer_warp, do_issue, lag, islot, iss, is]() {
            if (producer_warp && do_issue) {
                if (tid == kProducer) {
                    if (lag == 2) bulk_wait_read_all_but_one();
                    else bulk_wait_read_all();
                }
                __syncwarp();
                start(iss.h, iss.b, islot, is);
            }
        };
        bool alive;
        if (valid) {
            alive = process(cur.h, cur.b, slot, s, ok, refill);
        } else {
            alive = !__syncthreads_or(!ok);
            if (alive) refill();
        }
        if (!alive) {
            if (tid == kProducer) {
                raise_error(p.err, STEPQ_ERR_TIMEOUT);
                // drain this CTA's copies still in flight (items n .. issued), with a bound
                const int last = n < lag ? S_n - 1 : n - 1 - lag + S_n;
                for (int m = n; m <= last; m++) {
                    if (first + m * G >= p.items) break;
                    mbar_wait(&bars[m % S_n], (uint32_t)(m / S_n) & 1u, p.wait_cycles);
                }
                bulk_wait_all();
            }
            return;
        }
        __syncthreads();                                 // the page in stage s is final
        if (tid == kProducer) {
            if (valid) {
                fence_async_smem();
                store(cur.h, slot, s);
            }
            bulk_commit();
        }
        cur = nxt;
        if (n >= lag) {
            iss.step(G, gq, gr, p.nb);
            if (++is == S_n) is = 0;
        }
        if (++s == S_n) {
            s = 0;
            parity ^= 1u;
        }
    }
    if (tid == kProducer) bulk_wait_all();
}

}  // namespace pipe
}  // namespace stepq
