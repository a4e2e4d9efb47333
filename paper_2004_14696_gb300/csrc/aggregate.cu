// Eqs. (3)-(4) fused with the gradient statistics of Sect. 3.1 in one pass over
// the received rows of G: masked column mean g_t, SGD step on w, and per-block
// pieces of sum_j ||g_j||^2, sum_{l,j} (G[j,l] - g_t[l])^2 and ||g_t||^2.
//
// HBM-bound: each received row is read once with 128-bit streaming loads and w
// is read and written once, so the algorithmic traffic is (k d + 2 d) * 4 bytes
// (+ d * 4 if g_t is stored).
//
// Work split.  The columns are cut into warp chunks of 32 lanes x VEC float4
// (128 * VEC columns); a persistent grid of warps walks the chunks.  A warp owns
// its chunk for all k received rows, so the column reductions stay in its lanes'
// registers: no shared memory and no block barrier in the streaming loop.  Rows
// are processed UNROLL at a time, and the next batch's 128-bit loads are issued
// before the current batch is reduced.
//
// With DBW_ALL_ROW_NORMS the rows the mask leaves out are read too, after the
// received ones, for their squared norms only (Sect. 3.1's statistics still use
// the received rows alone); that adds (n - k) d * 4 bytes.  It is a separate
// instantiation of the kernel, so the default one is unchanged.
//
// Numerics.  Per column the warp keeps s1 = sum (x - c) and s2 = sum (x - c)^2 in
// fp32 with the shift c = the column's value in the first received row, so that
// sum_j (x_j - mean)^2 = s2 - s1^2 / k does not cancel.  Per-row squared norms
// are reduced across the warp in fp32 per chunk and accumulated in fp64 in shared
// memory (each row slot is owned by one warp, so no atomics); the column
// statistics are accumulated in fp64 per lane.  All reductions run in a fixed
// order, so results are deterministic for a given device.
#include "common.cuh"

namespace dbw {

namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int VEC = 2;      // float4 per lane per row: chunk = 32 * VEC * 4 = 256 columns
constexpr int UNROLL = 2;   // rows per batch; two batches in flight per lane
constexpr int kChunkCols = 32 * VEC * 4;

__device__ __forceinline__ float4 ldg_stream(const float4* p) {
    float4 v;
    asm volatile("ld.global.nc.L1::no_allocate.L2::256B.v4.f32 {%0,%1,%2,%3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "l"(p));
    return v;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// kAllRows: also the squared norms of the rows the mask leaves out (DBW_ALL_ROW_NORMS).
template <bool kAllRows>
__global__ void __launch_bounds__(kThreads, 3) aggregate_kernel(
    const float* __restrict__ G, int64_t ld, int n, int64_t d, const uint8_t* __restrict__ mask,
    float lr, float* __restrict__ w, float* __restrict__ gbar, double* __restrict__ partials,
    int nblocks) {
    extern __shared__ double smem_d[];
    double* rowacc = smem_d;                           // [kWarps][n] fp64 row-norm pieces
    // [n] rows in reading order: the received ones, then (kAllRows) the others
    int* sel = reinterpret_cast<int*>(smem_d + (size_t)kWarps * n);
    __shared__ int k_s;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) {
        int k = 0;
        for (int j = 0; j < n; ++j)
            if (mask[j]) sel[k++] = j;
        k_s = k;
        if (kAllRows) {
            int r = k;
            for (int j = 0; j < n; ++j)
                if (!mask[j]) sel[r++] = j;
        }
    }
    for (int i = tid; i < kWarps * n; i += kThreads) rowacc[i] = 0.0;
    __syncthreads();
    const int k = k_s;
    const int64_t hdr_flags = kAllRows ? DBW_ALL_ROW_NORMS : 0;
    if (k == 0) {   // nothing received: leave w untouched, record empty pieces
        double* vals = partials + kPartialsHeader + (n + 2);
        for (int q = tid; q < n + 2; q += kThreads) vals[(int64_t)q * nblocks + blockIdx.x] = 0.0;
        if (blockIdx.x == 0 && tid == 0) {
            int64_t* hdr = reinterpret_cast<int64_t*>(partials);
            hdr[0] = kPartialsMagic;
            hdr[1] = nblocks;
            hdr[2] = n;
            hdr[3] = hdr_flags;
        }
        return;
    }
    // rows read per chunk: the k received ones (their statistics), then with kAllRows
    // the n - k others (their squared norms only)
    const int nrows = kAllRows ? n : k;
    const float inv_k = 1.0f / (float)k;
    double* myrow = rowacc + (size_t)warp * n;

    double ss_acc = 0.0, g2_acc = 0.0;
    const int64_t nchunks = (d + kChunkCols - 1) / kChunkCols;
    const int64_t gwarp = (int64_t)blockIdx.x * kWarps + warp;
    const int64_t nwarps_total = (int64_t)nblocks * kWarps;

    for (int64_t chunk = gwarp; chunk < nchunks; chunk += nwarps_total) {
        const int64_t col0 = chunk * kChunkCols + lane * 4;
        // columns of this lane: col0 + v * 128 .. +3, v < VEC
        bool inb[VEC];
#pragma unroll
        for (int v = 0; v < VEC; ++v) inb[v] = (col0 + v * 128) < d;

        float4 c[VEC], s1[VEC], s2[VEC];
#pragma unroll
        for (int v = 0; v < VEC; ++v) {
            s1[v] = make_float4(0.f, 0.f, 0.f, 0.f);
            s2[v] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
        // row 0 of the received set gives the shift
        {
            const float* rowp = G + (int64_t)sel[0] * ld;
            float rn = 0.f;
#pragma unroll
            for (int v = 0; v < VEC; ++v) {
                const int64_t col = col0 + v * 128;
                float4 x = inb[v] ? ldg_stream(reinterpret_cast<const float4*>(rowp + col))
                                  : make_float4(0.f, 0.f, 0.f, 0.f);
                if (col + 3 >= d) {   // ragged tail inside the float4: zero columns >= d
                    if (col + 1 >= d) x.y = 0.f;
                    if (col + 2 >= d) x.z = 0.f;
                    if (col + 3 >= d) x.w = 0.f;
                }
                c[v] = x;
                rn += x.x * x.x + x.y * x.y + x.z * x.z + x.w * x.w;
            }
            rn = warp_sum(rn);
            if (lane == 0) myrow[0] += (double)rn;
        }
        // rows 1 .. k-1 in batches of UNROLL; the next batch's loads are in flight while
        // this batch is reduced
        float4 xn[UNROLL][VEC];
#pragma unroll
        for (int u = 0; u < UNROLL; ++u) {
            const int p = 1 + u;
            const float* rowp = G + (int64_t)sel[p < nrows ? p : 0] * ld;
#pragma unroll
            for (int v = 0; v < VEC; ++v) {
                const int64_t col = col0 + v * 128;
                xn[u][v] = (p < nrows && inb[v]) ? ldg_stream(reinterpret_cast<const float4*>(rowp + col))
                                                 : c[v];
            }
        }
        for (int p0 = 1; p0 < nrows; p0 += UNROLL) {
            float4 x[UNROLL][VEC];
#pragma unroll
            for (int u = 0; u < UNROLL; ++u)
#pragma unroll
                for (int v = 0; v < VEC; ++v) x[u][v] = xn[u][v];
            if (p0 + UNROLL < nrows) {
#pragma unroll
                for (int u = 0; u < UNROLL; ++u) {
                    const int p = p0 + UNROLL + u;
                    const float* rowp = G + (int64_t)sel[p < nrows ? p : 0] * ld;
#pragma unroll
                    for (int v = 0; v < VEC; ++v) {
                        const int64_t col = col0 + v * 128;
                        xn[u][v] = (p < nrows && inb[v])
                                       ? ldg_stream(reinterpret_cast<const float4*>(rowp + col))
                                       : c[v];
                    }
                }
            }
#pragma unroll
            for (int u = 0; u < UNROLL; ++u) {
                const int p = p0 + u;
                float rn = 0.f;
#pragma unroll
                for (int v = 0; v < VEC; ++v) {
                    float4 xv = x[u][v];
                    const int64_t col = col0 + v * 128;
                    if (col + 3 >= d) {
                        if (col + 1 >= d) xv.y = c[v].y;
                        if (col + 2 >= d) xv.z = c[v].z;
                        if (col + 3 >= d) xv.w = c[v].w;
                    }
                    if (!kAllRows || p < k) {   // rows read past the received ones add no statistics
                        const float dx0 = xv.x - c[v].x, dx1 = xv.y - c[v].y;
                        const float dx2 = xv.z - c[v].z, dx3 = xv.w - c[v].w;
                        s1[v].x += dx0; s1[v].y += dx1; s1[v].z += dx2; s1[v].w += dx3;
                        s2[v].x = fmaf(dx0, dx0, s2[v].x); s2[v].y = fmaf(dx1, dx1, s2[v].y);
                        s2[v].z = fmaf(dx2, dx2, s2[v].z); s2[v].w = fmaf(dx3, dx3, s2[v].w);
                    }
                    rn = fmaf(xv.x, xv.x, rn); rn = fmaf(xv.y, xv.y, rn);
                    rn = fmaf(xv.z, xv.z, rn); rn = fmaf(xv.w, xv.w, rn);
                }
                rn = warp_sum(rn);
                if (p < nrows && lane == 0) myrow[p] += (double)rn;
            }
        }
        // column epilogue: mean, SGD step, deviation sum, ||g_t||^2
        float ss_chunk = 0.f, g2_chunk = 0.f;
#pragma unroll
        for (int v = 0; v < VEC; ++v) {
            if (!inb[v]) continue;
            const int64_t col = col0 + v * 128;
            float m[4], dev[4];
            const float* c4 = &c[v].x;
            const float* a4 = &s1[v].x;
            const float* b4 = &s2[v].x;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                m[e] = c4[e] + a4[e] * inv_k;
                dev[e] = b4[e] - a4[e] * a4[e] * inv_k;
            }
            if (col + 3 < d) {
                float4 wv = *reinterpret_cast<const float4*>(w + col);
                wv.x = fmaf(-lr, m[0], wv.x); wv.y = fmaf(-lr, m[1], wv.y);
                wv.z = fmaf(-lr, m[2], wv.z); wv.w = fmaf(-lr, m[3], wv.w);
                *reinterpret_cast<float4*>(w + col) = wv;
                if (gbar) *reinterpret_cast<float4*>(gbar + col) = make_float4(m[0], m[1], m[2], m[3]);
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    ss_chunk += dev[e];
                    g2_chunk = fmaf(m[e], m[e], g2_chunk);
                }
            } else {
                for (int e = 0; e < 4 && col + e < d; ++e) {
                    w[col + e] = fmaf(-lr, m[e], w[col + e]);
                    if (gbar) gbar[col + e] = m[e];
                    ss_chunk += dev[e];
                    g2_chunk = fmaf(m[e], m[e], g2_chunk);
                }
            }
        }
        ss_acc += (double)ss_chunk;
        g2_acc += (double)g2_chunk;
    }

    // block partials: fixed-order reductions
    ss_acc = warp_sum_d(ss_acc);
    g2_acc = warp_sum_d(g2_acc);
    __shared__ double red[2][kWarps];
    if (lane == 0) {
        red[0][warp] = ss_acc;
        red[1][warp] = g2_acc;
    }
    __syncthreads();
    double* vals = partials + kPartialsHeader + (n + 2);
    for (int q = tid; q < n; q += kThreads) vals[(int64_t)q * nblocks + blockIdx.x] = 0.0;
    __syncthreads();
    // rows are indexed by reading position in rowacc; scatter them to worker ids
    for (int p = tid; p < nrows; p += kThreads) {
        double s = 0.0;
        for (int wv = 0; wv < kWarps; ++wv) s += rowacc[(size_t)wv * n + p];
        vals[(int64_t)sel[p] * nblocks + blockIdx.x] = s;
    }
    if (tid == 0) {
        double a = 0.0, b = 0.0;
        for (int wv = 0; wv < kWarps; ++wv) {
            a += red[0][wv];
            b += red[1][wv];
        }
        vals[(int64_t)n * nblocks + blockIdx.x] = a;
        vals[(int64_t)(n + 1) * nblocks + blockIdx.x] = b;
        if (blockIdx.x == 0) {
            int64_t* hdr = reinterpret_cast<int64_t*>(partials);
            hdr[0] = kPartialsMagic;
            hdr[1] = nblocks;
            hdr[2] = n;
            hdr[3] = hdr_flags;
        }
    }
}

size_t agg_smem_bytes(int n) { return (size_t)kWarps * n * sizeof(double) + (size_t)n * sizeof(int); }

}  // namespace

AggGeometry agg_geometry(int n, int64_t d) {
    AggGeometry g;
    int per_sm = 0;
    // both instantiations have the same launch shape; the default one sets the grid
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, aggregate_kernel<false>, kThreads, agg_smem_bytes(n));
    if (per_sm < 1) per_sm = 1;
    const int64_t nchunks = (d + kChunkCols - 1) / kChunkCols;
    int64_t blocks = (int64_t)sm_count() * per_sm;
    const int64_t need = (nchunks + kWarps - 1) / kWarps;
    if (blocks > need) blocks = need;
    if (blocks < 1) blocks = 1;
    g.blocks = (int)blocks;
    g.rows_stride = n + 2;
    g.bytes = (size_t)kPartialsHeader * sizeof(int64_t) + (size_t)(n + 2) * (blocks + 1) * sizeof(double);
    return g;
}

namespace {
template <bool kAllRows>
cudaError_t launch_aggregate_t(const float* G, int64_t ld, int n, int64_t d, const uint8_t* mask, float lr,
                               float* w, float* gbar, double* partials, const AggGeometry& g, cudaStream_t st) {
    const size_t smem = agg_smem_bytes(n);
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(aggregate_kernel<kAllRows>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    aggregate_kernel<kAllRows><<<g.blocks, kThreads, smem, st>>>(G, ld, n, d, mask, lr, w, gbar, partials,
                                                                 g.blocks);
    return cudaGetLastError();
}
}  // namespace

cudaError_t launch_aggregate(const float* G, int64_t ld, int n, int64_t d, const uint8_t* mask,
                             float lr, float* w, float* gbar, int flags, double* partials, const AggGeometry& g,
                             cudaStream_t st) {
    if (flags & DBW_ALL_ROW_NORMS)
        return launch_aggregate_t<true>(G, ld, n, d, mask, lr, w, gbar, partials, g, st);
    return launch_aggregate_t<false>(G, ld, n, d, mask, lr, w, gbar, partials, g, st);
}

}  // namespace dbw
