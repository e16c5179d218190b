// COO -> CSR grouped by target node: the "reduce by key" grouping of the
// graph map-reduce framework (tf_geometric Section 2.1.2, Fig. 5b), with the
// target node as the key.
//
// Method: a stable least-significant-digit radix sort of the edges by target
// id, one pass per digit of ceil(log2 N) bits split into <= 10-bit digits.
// Each pass is reduce-then-scan over 4096-edge tiles:
//   upsweep   per-tile digit histogram -> cnt[digit][tile] (digit-major)
//   scan      exclusive scan of cnt in that order: offs[digit][tile] = (edges
//             of all smaller digits) + (edges of this digit in earlier tiles),
//             the first output slot of every (tile, digit) run; taking the
//             tiles in order inside a digit keeps the sort stable
//   downsweep ranks each tile's elements in original order, stages the tile
//             in shared memory in digit order and writes each digit's run
//             with coalesced stores
// No kernel waits on another CTA, so nothing can spin.  The first pass reads
// the int64 edge_index directly and checks every id; the last pass writes
// col (source) and perm (original edge id) in final order, plus the sorted
// keys from which rowptr is found by binary search.
#include <type_traits>

#include "common.cuh"

namespace tfg {
namespace {

constexpr int kTile = 4096;                       // edges per CTA tile
constexpr int kMaxDigitBits = 10;
constexpr int kUpThreads = 256;
constexpr int kScanThreads = 256;
constexpr int kScanItems = 16;
constexpr int kScanChunk = kScanThreads * kScanItems;

struct SortPlan {
    int passes;
    int width;
};

SortPlan plan_for(int64_t n) {
    int bits = 1;
    while ((int64_t(1) << bits) < n) ++bits;
    int passes = (bits + kMaxDigitBits - 1) / kMaxDigitBits;
    int width = (bits + passes - 1) / passes;
    return {passes, width};
}

size_t align256(size_t b) { return (b + 255) & ~size_t(255); }

// An id outside [0, n) is reported and replaced by 0, so every later index
// stays in bounds.  The upsweep and downsweep clamp identically, keeping the
// per-tile counts consistent with the ranks.
__device__ __forceinline__ uint32_t checked_id(int64_t v, int64_t n, int32_t *status) {
    if (v < 0 || v >= n) {
        if (status) set_status(status, TFG_ERR_INDEX_RANGE);
        return 0u;
    }
    return static_cast<uint32_t>(v);
}

// IdT: the element type of the caller's edge_index (int64, or int32 for
// tfg_build_csr32); only the first pass reads it.
template <bool FIRST, typename IdT = int64_t>
__global__ void __launch_bounds__(kUpThreads)
radix_upsweep(const IdT *__restrict__ dst64, const uint32_t *__restrict__ key32, int64_t e,
              int64_t n, int shift, int width, int num_tiles, int32_t *__restrict__ cnt,
              int32_t *status) {
    extern __shared__ int32_t s_cnt[];
    const int radix = 1 << width;
    for (int d = threadIdx.x; d < radix; d += kUpThreads) s_cnt[d] = 0;
    __syncthreads();
    const int64_t base = static_cast<int64_t>(blockIdx.x) * kTile;
    const int64_t stop = min64(e, base + kTile);
    for (int64_t i = base + threadIdx.x; i < stop; i += kUpThreads) {
        uint32_t key = FIRST ? checked_id(__ldg(dst64 + i), n, status) : __ldg(key32 + i);
        atomicAdd(&s_cnt[(key >> shift) & (radix - 1)], 1);
    }
    __syncthreads();
    for (int d = threadIdx.x; d < radix; d += kUpThreads)
        cnt[static_cast<int64_t>(d) * num_tiles + blockIdx.x] = s_cnt[d];
}

// ---- exclusive scan of an int32 array (in place), three kernels ----------
__device__ int32_t block_exclusive_scan(int32_t v, int32_t *total) {
    __shared__ int32_t warp_sums[kScanThreads / 32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int32_t incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int32_t y = __shfl_up_sync(kFull, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) warp_sums[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        const int32_t s = lane < kScanThreads / 32 ? warp_sums[lane] : 0;
        int32_t si = s;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int32_t y = __shfl_up_sync(kFull, si, o);
            if (lane >= o) si += y;
        }
        if (lane < kScanThreads / 32) warp_sums[lane] = si - s;
        if (lane == kScanThreads / 32 - 1 && total) *total = si;
    }
    __syncthreads();
    const int32_t r = incl - v + warp_sums[warp];
    __syncthreads();
    return r;
}

__global__ void __launch_bounds__(kScanThreads)
scan_reduce(const int32_t *__restrict__ data, int64_t m, int32_t *__restrict__ sums) {
    const int64_t base = static_cast<int64_t>(blockIdx.x) * kScanChunk;
    int32_t s = 0;
#pragma unroll
    for (int i = 0; i < kScanItems; ++i) {
        const int64_t k = base + i * kScanThreads + threadIdx.x;
        if (k < m) s += data[k];
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(kFull, s, o);
    __shared__ int32_t ws[kScanThreads / 32];
    if ((threadIdx.x & 31) == 0) ws[threadIdx.x >> 5] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
        int32_t t = 0;
        for (int w = 0; w < kScanThreads / 32; ++w) t += ws[w];
        sums[blockIdx.x] = t;
    }
}

__global__ void __launch_bounds__(kScanThreads) scan_top(int32_t *sums, int nb) {
    __shared__ int32_t carry;
    __shared__ int32_t tot;
    if (threadIdx.x == 0) carry = 0;
    __syncthreads();
    for (int base = 0; base < nb; base += kScanThreads) {
        const int k = base + threadIdx.x;
        const int32_t v = k < nb ? sums[k] : 0;
        const int32_t ex = block_exclusive_scan(v, &tot);
        if (k < nb) sums[k] = ex + carry;
        __syncthreads();
        if (threadIdx.x == 0) carry += tot;
        __syncthreads();
    }
}

// Each thread scans kScanItems consecutive values; loads are staged through
// shared memory so the global reads and writes stay coalesced.
__global__ void __launch_bounds__(kScanThreads)
scan_down(int32_t *data, int64_t m, const int32_t *__restrict__ sums) {
    __shared__ int32_t s_v[kScanChunk + kScanChunk / 32];   // padded against bank conflicts
    const int64_t base = static_cast<int64_t>(blockIdx.x) * kScanChunk;
    auto at = [](int i) { return i + (i >> 5); };
#pragma unroll
    for (int i = 0; i < kScanItems; ++i) {
        const int j = i * kScanThreads + threadIdx.x;
        s_v[at(j)] = base + j < m ? data[base + j] : 0;
    }
    __syncthreads();
    int32_t v[kScanItems];
    int32_t local = 0;
#pragma unroll
    for (int i = 0; i < kScanItems; ++i) {
        v[i] = s_v[at(threadIdx.x * kScanItems + i)];
        local += v[i];
    }
    int32_t run = block_exclusive_scan(local, nullptr) + sums[blockIdx.x];
#pragma unroll
    for (int i = 0; i < kScanItems; ++i) {
        s_v[at(threadIdx.x * kScanItems + i)] = run;
        run += v[i];
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < kScanItems; ++i) {
        const int j = i * kScanThreads + threadIdx.x;
        if (base + j < m) data[base + j] = s_v[at(j)];
    }
}

cudaError_t exclusive_scan(int32_t *data, int64_t m, int32_t *sums, cudaStream_t s) {
    const int nb = ceil_div(m, kScanChunk);
    scan_reduce<<<nb, kScanThreads, 0, s>>>(data, m, sums);
    scan_top<<<1, kScanThreads, 0, s>>>(sums, nb);
    scan_down<<<nb, kScanThreads, 0, s>>>(data, m, sums);
    return cudaGetLastError();
}

// ---- downsweep ------------------------------------------------------------
// 16 warps share one 4096-edge tile, 8 elements per lane.  Every global load
// of the tile is issued up front, so the tile waits on memory once.
//   A  per round of 32 elements, lanes holding equal digits are found with
//      one ballot per digit bit; the group's leader advances the warp's
//      private counter of that digit, and each element keeps its rank among
//      the warp's elements of its digit so far (a byte, 8 per lane packed in
//      two registers)
//   B  per digit: warp-major exclusive prefix and tile total; block scan of
//      the totals over digits -> each digit's first slot in the tile; per
//      digit, global base minus tile start
//   C  stable slot = digit's first tile slot + warp prefix + rank; key,
//      source and edge id are staged in three arrays
//   D  the tile leaves in digit order, consecutive threads writing
//      consecutive positions of each digit's run
#ifndef TFG_DS_FULL_TILES
#define TFG_DS_FULL_TILES 1   // separate code for full tiles (no bounds tests)
#endif
constexpr bool kDsFullTiles = TFG_DS_FULL_TILES != 0;
constexpr int kDsWarps = 16;
constexpr int kDsThreads = kDsWarps * 32;
constexpr int kDsItems = kTile / kDsThreads;   // 8 per lane

size_t downsweep_smem(int radix) {
    return sizeof(uint32_t) * 3 * kTile + sizeof(int32_t) * kDsWarps * radix +
           sizeof(int32_t) * 2 * radix + sizeof(int32_t) * 32;
}

// Lanes of the warp whose value of dig equals this lane's, for dig below
// 2^bits: one ballot per bit (measured faster here than __match_any_sync).
__device__ __forceinline__ unsigned peers_from_bit(unsigned peers, uint32_t dig, int b) {
    const bool set = (dig >> b) & 1u;
    const unsigned bal = __ballot_sync(kFull, set);
    return peers & (set ? bal : ~bal);
}

template <int BITS>   // bit count known at compile time: the loop unrolls
__device__ __forceinline__ unsigned same_digit_lanes(uint32_t dig) {
    unsigned peers = kFull;
#pragma unroll
    for (int b = 0; b < BITS; ++b) peers = peers_from_bit(peers, dig, b);
    return peers;
}

__device__ __forceinline__ unsigned same_digit_lanes(uint32_t dig, int bits) {
    unsigned peers = kFull;
#pragma unroll 1
    for (int b = 0; b < bits; ++b) peers = peers_from_bit(peers, dig, b);
    return peers;
}

// W > 0 fixes the digit width at compile time (the ballot loop unrolls and
// the per-digit loops get constant bounds); W = 0 takes it from width_arg.
template <bool FIRST, int W, typename IdT = int64_t>
__global__ void __launch_bounds__(kDsThreads, 2)
radix_downsweep(const IdT *__restrict__ src64, const IdT *__restrict__ dst64,
                const uint32_t *__restrict__ key_in, const int32_t *__restrict__ src_in,
                const int32_t *__restrict__ eid_in, int64_t e, int64_t n, int shift,
                int width_arg, int num_tiles, const int32_t *__restrict__ offs,
                uint32_t *__restrict__ key_out, int32_t *__restrict__ src_out,
                int32_t *__restrict__ eid_out, int32_t *status) {
    extern __shared__ __align__(16) unsigned char smem[];
    const int width = W > 0 ? W : width_arg;
    const int radix = 1 << width;
    uint32_t *s_key = reinterpret_cast<uint32_t *>(smem);                 // [tile]
    int32_t *s_src = reinterpret_cast<int32_t *>(s_key + kTile);           // [tile]
    int32_t *s_eid = s_src + kTile;                                        // [tile]
    int32_t *s_cnt = s_eid + kTile;                                        // [warp][digit]
    int32_t *s_tstart = s_cnt + kDsWarps * radix;                          // [digit]
    int32_t *s_delta = s_tstart + radix;                                   // [digit]
    int32_t *s_chunk = s_delta + radix;                                    // [32]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t tile0 = static_cast<int64_t>(blockIdx.x) * kTile;
    const int count = static_cast<int>(min64(kTile, e - tile0));
    // every tile but the last is full: its copy of the code has no bounds tests
    auto run = [&](auto full_tag) {
        constexpr bool FULL = decltype(full_tag)::value;
        int32_t *mine = s_cnt + warp * radix;
        for (int d = lane; d < radix; d += 32) mine[d] = 0;
        for (int d = threadIdx.x; d < radix; d += kDsThreads)
            s_delta[d] = offs[static_cast<int64_t>(d) * num_tiles + blockIdx.x];   // global base for now

        // All loads of this warp's sub-tile, issued together.
        const int64_t wbase = tile0 + static_cast<int64_t>(warp) * 32 * kDsItems;
        uint32_t keys[kDsItems];
        int32_t srcs[kDsItems], eids[kDsItems];
    #pragma unroll
        for (int r = 0; r < kDsItems; ++r) {
            const int64_t idx = wbase + r * 32 + lane;
            keys[r] = 0;
            srcs[r] = 0;
            eids[r] = 0;
            if (FULL || idx < e) {
                if (FIRST) {
                    keys[r] = checked_id(__ldg(dst64 + idx), n, nullptr);
                    srcs[r] = static_cast<int32_t>(checked_id(__ldg(src64 + idx), n, status));
                    eids[r] = static_cast<int32_t>(idx);
                } else {
                    keys[r] = __ldg(key_in + idx);
                    srcs[r] = __ldg(src_in + idx);
                    eids[r] = __ldg(eid_in + idx);
                }
            }
        }
        __syncwarp();

        const unsigned lower = (1u << lane) - 1u;
        // A: per-warp digit counts, and each element's rank among the warp's
        // earlier elements of its digit (one leader per digit group bumps the
        // warp's private counter)
        uint32_t rank_lo = 0, rank_hi = 0;   // 8 ranks < 256, one byte each
    #pragma unroll
        for (int r = 0; r < kDsItems; ++r) {
            const bool ok = FULL || wbase + r * 32 + lane < e;
            const uint32_t dig = ok ? ((keys[r] >> shift) & (radix - 1)) : uint32_t(radix);
            // a partial tile marks its missing elements with digit radix: one bit more
            unsigned peers;
            if constexpr (W > 0) peers = same_digit_lanes<FULL ? W : W + 1>(dig);
            else peers = same_digit_lanes(dig, FULL ? width : width + 1);
            const int leader = __ffs(peers) - 1;
            int32_t base = 0;
            if (ok && lane == leader) {
                base = mine[dig];
                mine[dig] = base + __popc(peers);
            }
            base = __shfl_sync(kFull, base, leader);
            const uint32_t rk = static_cast<uint32_t>(base + __popc(peers & lower));
            if (r < 4) rank_lo |= rk << (8 * r);
            else rank_hi |= rk << (8 * (r - 4));
            __syncwarp();
        }
        __syncthreads();

        // B: warp-major prefix per digit, tile totals, then a block scan over digits.
        for (int d = threadIdx.x; d < radix; d += kDsThreads) {
            int32_t c[kDsWarps];
    #pragma unroll
            for (int w = 0; w < kDsWarps; ++w) c[w] = s_cnt[w * radix + d];
            int32_t run = 0;
    #pragma unroll
            for (int w = 0; w < kDsWarps; ++w) {
                s_cnt[w * radix + d] = run;
                run += c[w];
            }
            s_tstart[d] = run;
        }
        __syncthreads();
        const int chunks = (radix + 31) / 32;   // <= 32
        for (int ch = warp; ch < chunks; ch += kDsWarps) {   // scan of each 32-digit chunk
            const int d = ch * 32 + lane;
            const int32_t v = d < radix ? s_tstart[d] : 0;
            int32_t incl = v;
    #pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int32_t y = __shfl_up_sync(kFull, incl, o);
                if (lane >= o) incl += y;
            }
            if (d < radix) s_tstart[d] = incl - v;
            if (lane == 31) s_chunk[ch] = incl;
        }
        __syncthreads();
        if (warp == 0) {   // exclusive scan of the chunk totals
            const int32_t v = lane < chunks ? s_chunk[lane] : 0;
            int32_t incl = v;
    #pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int32_t y = __shfl_up_sync(kFull, incl, o);
                if (lane >= o) incl += y;
            }
            if (lane < chunks) s_chunk[lane] = incl - v;
        }
        __syncthreads();
        for (int d = threadIdx.x; d < radix; d += kDsThreads) {
            const int32_t ts = s_tstart[d] + s_chunk[d >> 5];
            s_tstart[d] = ts;   // first tile slot of digit d
            s_delta[d] -= ts;   // global position of tile slot i of digit d = delta[d] + i
        }
        __syncthreads();

        // C: stable slot of every element; stage (key, source, edge id).
    #pragma unroll
        for (int r = 0; r < kDsItems; ++r) {
            const bool ok = FULL || wbase + r * 32 + lane < e;
            const uint32_t dig = ok ? ((keys[r] >> shift) & (radix - 1)) : uint32_t(radix);
            if (ok) {
                const uint32_t rk = (r < 4 ? rank_lo >> (8 * r) : rank_hi >> (8 * (r - 4))) & 0xffu;
                const int slot = mine[dig] + s_tstart[dig] + static_cast<int>(rk);
                s_key[slot] = keys[r];
                s_src[slot] = srcs[r];
                s_eid[slot] = eids[r];
            }
        }
        __syncthreads();

        // D: write the tile out, one coalesced run per digit.
    #pragma unroll
        for (int j = 0; j < kDsItems; ++j) {
            const int i = threadIdx.x + j * kDsThreads;
            if (FULL || i < count) {
                const uint32_t k = s_key[i];
                const int d = static_cast<int>((k >> shift) & (radix - 1));
                const int64_t pos = static_cast<int64_t>(s_delta[d]) + i;
                key_out[pos] = k;
                src_out[pos] = s_src[i];
                eid_out[pos] = s_eid[i];
            }
        }
    };
    if (kDsFullTiles && count == kTile) run(std::true_type{});
    else run(std::false_type{});
}

// rowptr[k] = first sorted position whose key is >= k, for k in [0, n].
__global__ void rowptr_from_sorted(const uint32_t *__restrict__ keys, int64_t e, int64_t n,
                                   int32_t *__restrict__ rowptr) {
    const int64_t k = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (k > n) return;
    int64_t lo = 0, hi = e;
    while (lo < hi) {
        const int64_t mid = (lo + hi) >> 1;
        if (static_cast<int64_t>(__ldg(keys + mid)) < k) lo = mid + 1;
        else hi = mid;
    }
    rowptr[k] = static_cast<int32_t>(lo);
}

__global__ void degree_from_rowptr(const int32_t *__restrict__ rowptr, int64_t n,
                                   int32_t *__restrict__ deg) {
    const int64_t t = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (t < n) deg[t] = rowptr[t + 1] - rowptr[t];
}

#ifndef TFG_DS_STATIC_WIDTH
#define TFG_DS_STATIC_WIDTH 1   // downsweeps with compile-time digit widths 6..10
#endif

template <typename IdT>
using DownsweepFn = void (*)(const IdT *, const IdT *, const uint32_t *, const int32_t *,
                             const int32_t *, int64_t, int64_t, int, int, int, const int32_t *,
                             uint32_t *, int32_t *, int32_t *, int32_t *);

// Every multi-pass plan has digits of 6..10 bits (plan_for), so those widths
// get their own code; single-pass sorts of small graphs take the generic one.
// Later passes read the library's own int32 arrays: they take IdT = int64_t
// (their edge_index pointers are null) whatever the caller's id type.
template <bool FIRST, typename IdT>
DownsweepFn<IdT> downsweep_for(int width) {
    switch (TFG_DS_STATIC_WIDTH ? width : 0) {
        case 6: return radix_downsweep<FIRST, 6, IdT>;
        case 7: return radix_downsweep<FIRST, 7, IdT>;
        case 8: return radix_downsweep<FIRST, 8, IdT>;
        case 9: return radix_downsweep<FIRST, 9, IdT>;
        case 10: return radix_downsweep<FIRST, 10, IdT>;
        default: return radix_downsweep<FIRST, 0, IdT>;
    }
}

}  // namespace

size_t csr_workspace_bytes(int64_t n, int64_t e) {
    if (e <= 0) return 256;
    const SortPlan p = plan_for(n);
    const int64_t tiles = ceil_div(e, kTile);
    const int64_t radix = int64_t(1) << p.width;
    const size_t a = align256(sizeof(int32_t) * 3 * size_t(e));
    const size_t b = align256(sizeof(int32_t) * (p.passes >= 3 ? 3 : 1) * size_t(e));
    const size_t h = align256(sizeof(int32_t) * size_t(radix * tiles));
    const size_t sums = align256(sizeof(int32_t) * size_t(ceil_div(radix * tiles, kScanChunk)));
    return a + b + h + sums;
}

namespace {
template <typename IdT>
cudaError_t build_csr_impl(const IdT *edge_index, int64_t e, int64_t n, int32_t *rowptr,
                           int32_t *col, int32_t *perm, int32_t *in_degree, void *ws,
                           int32_t *status, cudaStream_t s, bool by_source) {
    cudaError_t err = cudaMemsetAsync(status, 0, sizeof(int32_t), s);
    if (err != cudaSuccess) return err;
    const uint32_t *sorted_keys = nullptr;
    if (e > 0) {
        const SortPlan p = plan_for(n);
        const int tiles = ceil_div(e, kTile);
        const int radix = 1 << p.width;
        char *w = static_cast<char *>(ws);
        struct Buf { uint32_t *key; int32_t *src; int32_t *eid; } buf[2];
        buf[0].key = reinterpret_cast<uint32_t *>(w);
        buf[0].src = reinterpret_cast<int32_t *>(buf[0].key + e);
        buf[0].eid = buf[0].src + e;
        w += align256(sizeof(int32_t) * 3 * size_t(e));
        buf[1].key = reinterpret_cast<uint32_t *>(w);
        buf[1].src = reinterpret_cast<int32_t *>(buf[1].key + e);
        buf[1].eid = buf[1].src + e;
        w += align256(sizeof(int32_t) * (p.passes >= 3 ? 3 : 1) * size_t(e));
        int32_t *cnt = reinterpret_cast<int32_t *>(w);
        w += align256(sizeof(int32_t) * size_t(int64_t(radix) * tiles));
        int32_t *sums = reinterpret_cast<int32_t *>(w);

        // the key row is row 1 (targets), or row 0 (sources) for the transposed CSR
        const IdT *src64 = by_source ? edge_index + e : edge_index;
        const IdT *dst64 = by_source ? edge_index : edge_index + e;
        const DownsweepFn<IdT> down_first = downsweep_for<true, IdT>(p.width);
        const DownsweepFn<int64_t> down_later = downsweep_for<false, int64_t>(p.width);
        // the limit is set to the largest tile any width needs, so concurrent
        // builds of different sizes never lower it under one another's launch
        const int smem_max = static_cast<int>(downsweep_smem(1 << kMaxDigitBits));
        err = cudaFuncSetAttribute(down_first, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_max);
        if (err == cudaSuccess)
            err = cudaFuncSetAttribute(down_later, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_max);
        if (err != cudaSuccess) return err;
        for (int pass = 0; pass < p.passes; ++pass) {
            const int shift = pass * p.width;
            const bool first = pass == 0, last = pass == p.passes - 1;
            const Buf &in = buf[(pass + 1) & 1];
            Buf out = buf[pass & 1];
            if (last) { out.src = col; out.eid = perm; }
            if (first)
                radix_upsweep<true, IdT><<<tiles, kUpThreads, radix * sizeof(int32_t), s>>>(
                    dst64, nullptr, e, n, shift, p.width, tiles, cnt, status);
            else
                radix_upsweep<false, int64_t><<<tiles, kUpThreads, radix * sizeof(int32_t), s>>>(
                    nullptr, in.key, e, n, shift, p.width, tiles, cnt, status);
            err = exclusive_scan(cnt, int64_t(radix) * tiles, sums, s);
            if (err != cudaSuccess) return err;
            const size_t smem = downsweep_smem(radix);
            if (first)
                down_first<<<tiles, kDsThreads, smem, s>>>(
                    src64, dst64, nullptr, nullptr, nullptr, e, n, shift, p.width, tiles, cnt,
                    out.key, out.src, out.eid, status);
            else
                down_later<<<tiles, kDsThreads, smem, s>>>(
                    nullptr, nullptr, in.key, in.src, in.eid, e, n, shift, p.width, tiles, cnt,
                    out.key, out.src, out.eid, status);
            err = cudaGetLastError();
            if (err != cudaSuccess) return err;
            sorted_keys = out.key;
        }
    }
    rowptr_from_sorted<<<ceil_div(n + 1, 256), 256, 0, s>>>(sorted_keys, e, n, rowptr);
    if (n > 0) degree_from_rowptr<<<ceil_div(n, 256), 256, 0, s>>>(rowptr, n, in_degree);
    return cudaGetLastError();
}
}  // namespace

cudaError_t launch_build_csr(const int64_t *edge_index, int64_t e, int64_t n, int32_t *rowptr,
                             int32_t *col, int32_t *perm, int32_t *in_degree, void *ws,
                             int32_t *status, cudaStream_t s, bool by_source) {
    return build_csr_impl(edge_index, e, n, rowptr, col, perm, in_degree, ws, status, s,
                          by_source);
}

cudaError_t launch_build_csr32(const int32_t *edge_index, int64_t e, int64_t n, int32_t *rowptr,
                               int32_t *col, int32_t *perm, int32_t *in_degree, void *ws,
                               int32_t *status, cudaStream_t s, bool by_source) {
    return build_csr_impl(edge_index, e, n, rowptr, col, perm, in_degree, ws, status, s,
                          by_source);
}

}  // namespace tfg
