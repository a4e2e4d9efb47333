// Eq. (2) for all n workers with bf16 GEMM operands on the tcgen05 tensor cores.
//
// Same computation as the SIMT pass in grads.cu (forward over the stacked
// M = n B rows, softmax cross entropy, backward with a per-worker weight
// gradient of depth K = B), laid out so that every GEMM has both operands
// K-major, which is what the tcgen05 kernel of gemm_tc.cu consumes:
//
//   forward   Z_l = A_{l-1} . W_l^T          A = act[l-1] [M, in],   B = W_l [out, in]
//   dX        dZ_{l-1} = dZ_l . W_l          A = dZ_l [M, out],      B = W_l^T [in, out]
//   dW        G_i = dZ_l[i]^T . A_{l-1}[i]   A = dZ_l^T [out, M],    B = A_{l-1}^T [in, M]
//                                            (worker i: columns i*B .. i*B+B-1, K = B)
//
// The transposed activations and dZ are written by the epilogue that produces
// them (a store whose 32 lanes cover 32 consecutive samples, 64 contiguous
// bytes), X^T and dZ_L^T by a tiled transpose, W^T by a tiled cast-transpose.
// Leading dimensions are padded to multiples of 8 elements (16 bytes, the TMA
// stride rule); padding is never read (tensor maps carry the logical extents).
#include <math.h>

#include "gemm_tc.cuh"
#include "grads.cuh"

namespace dbw {

namespace {

inline int64_t rup(int64_t x, int64_t m) { return (x + m - 1) / m * m; }

// One pass over fp32 rows: out[m, :] = bf16(src[row(m), :]) and outT = its
// transpose, for m < rows (cols logical columns; padding is never written).  A
// CTA handles a 64 x 64 tile: the rows are read as float4 where aligned, the
// bf16 tile is written row-major with 8-byte stores and, through a padded
// shared-memory tile, column-major with 8-byte stores along m.  row(m) < 0 makes
// row m zero.  Used for X (gathered minibatch rows) and for W_l (rows = out).
template <class RowMap>
__device__ __forceinline__ void cast_transpose_tile(const float* __restrict__ src, int64_t lds, int rows, int cols,
                                                    RowMap rowmap, __nv_bfloat16* __restrict__ out, int64_t ldo,
                                                    __nv_bfloat16* __restrict__ outT, int64_t ldT, int c0, int m0) {
    __shared__ __nv_bfloat16 tile[64][64 + 8];
    const int live = rowmap.live(rows);
    if (m0 >= live) return;
    const int t = threadIdx.x;
    // all four rows' loads first, so that each thread has 64 bytes in flight
    float v[4][4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int e = t + 256 * q;
        const int r = e >> 4, c = c0 + 4 * (e & 15);
        const int m = m0 + r;
#pragma unroll
        for (int j = 0; j < 4; ++j) v[q][j] = 0.f;
        if (m < live && c < cols) {
            const int64_t sr = rowmap(m);
            if (sr >= 0) {
                const float* p = src + sr * lds + c;
                if (c + 3 < cols && ((reinterpret_cast<uintptr_t>(p) & 15u) == 0)) {
                    const float4 f = __ldcs(reinterpret_cast<const float4*>(p));
                    v[q][0] = f.x, v[q][1] = f.y, v[q][2] = f.z, v[q][3] = f.w;
                } else {
                    for (int j = 0; j < 4 && c + j < cols; ++j) v[q][j] = p[j];
                }
            }
        }
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int e = t + 256 * q;
        const int r = e >> 4, c = c0 + 4 * (e & 15);
        const int m = m0 + r;
        __nv_bfloat16 h[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) h[j] = __float2bfloat16_rn(v[q][j]);
#pragma unroll
        for (int j = 0; j < 4; ++j) tile[r][4 * (e & 15) + j] = h[j];
        if (m < live && c < cols) {
            __nv_bfloat16* o = out + static_cast<int64_t>(m) * ldo + c;
            if (c + 3 < cols && ((reinterpret_cast<uintptr_t>(o) & 7u) == 0)) {
                uint2 pk;
                pk.x = static_cast<uint32_t>(__bfloat16_as_ushort(h[0])) |
                       (static_cast<uint32_t>(__bfloat16_as_ushort(h[1])) << 16);
                pk.y = static_cast<uint32_t>(__bfloat16_as_ushort(h[2])) |
                       (static_cast<uint32_t>(__bfloat16_as_ushort(h[3])) << 16);
                *reinterpret_cast<uint2*>(o) = pk;
            } else {
                for (int j = 0; j < 4 && c + j < cols; ++j) o[j] = h[j];
            }
        }
    }
    __syncthreads();
    if (!outT) return;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int e = t + 256 * q;
        const int cc = e >> 4, r = 4 * (e & 15);
        const int c = c0 + cc, m = m0 + r;
        if (c >= cols || m >= live) continue;
        __nv_bfloat16* o = outT + static_cast<int64_t>(c) * ldT + m;
        if (m + 3 < live && ((reinterpret_cast<uintptr_t>(o) & 7u) == 0)) {
            uint2 pk;
            pk.x = static_cast<uint32_t>(__bfloat16_as_ushort(tile[r][cc])) |
                   (static_cast<uint32_t>(__bfloat16_as_ushort(tile[r + 1][cc])) << 16);
            pk.y = static_cast<uint32_t>(__bfloat16_as_ushort(tile[r + 2][cc])) |
                   (static_cast<uint32_t>(__bfloat16_as_ushort(tile[r + 3][cc])) << 16);
            *reinterpret_cast<uint2*>(o) = pk;
        } else {
            for (int j = 0; j < 4 && m + j < live; ++j) o[j] = tile[r + j][cc];
        }
    }
}

template <class RowMap>
__global__ void __launch_bounds__(256) cast_transpose_tile_kernel(const float* __restrict__ src, int64_t lds,
                                                                  int rows, int cols, RowMap rowmap,
                                                                  __nv_bfloat16* __restrict__ out, int64_t ldo,
                                                                  __nv_bfloat16* __restrict__ outT, int64_t ldT) {
    cast_transpose_tile(src, lds, rows, cols, rowmap, out, ldo, outT, ldT, blockIdx.x * 64, blockIdx.y * 64);
}

// Row maps of cast_transpose_tile_kernel.
struct IdentityRows {   // W_l: row o of the matrix
    __device__ int live(int rows) const { return rows; }
    __device__ int64_t operator()(int m) const { return m; }
};
// Every layer's W_l -> bf16 W_l and W_l^T in one launch: the layers' 64 x 64 tiles one
// after the other in x (t0: first tile of layer l; tx: its tiles per row of tiles).
struct WeightCasts {
    int L;
    const float* w[DBW_LMAX];
    int fin[DBW_LMAX], fout[DBW_LMAX], tx[DBW_LMAX];
    int t0[DBW_LMAX + 1];
    __nv_bfloat16* wb[DBW_LMAX];
    int64_t ldw[DBW_LMAX];
    __nv_bfloat16* wt[DBW_LMAX];
    int64_t ldwt[DBW_LMAX];
};

__global__ void __launch_bounds__(256) cast_transpose_weights_kernel(WeightCasts a) {
    int l = 0;
    while (l + 1 < a.L && static_cast<int>(blockIdx.x) >= a.t0[l + 1]) ++l;
    const int t = blockIdx.x - a.t0[l];
    cast_transpose_tile(a.w[l], a.fin[l], a.fout[l], a.fin[l], IdentityRows{}, a.wb[l], a.ldw[l], a.wt[l], a.ldwt[l],
                        (t % a.tx[l]) * 64, (t / a.tx[l]) * 64);
}

struct GatherRows {     // X of the per-worker pass: pool row idx[m]; an index outside [0, S) reads row 0
    const int32_t* idx;
    int64_t S;
    __device__ int live(int rows) const { return rows; }
    __device__ int64_t operator()(int m) const {
        const int64_t r = idx[m];
        return (r < 0 || r >= S) ? 0 : r;
    }
};

// Rows of the stacked buffers that a received-workers pass computes: the k B
// received rows rounded up to the 128-row GEMM tile (all M when kdev is null).
__device__ __forceinline__ int live_rows(const int* kdev, int B, int M) {
    if (!kdev) return M;
    const int k = *kdev;
    const long long r = (static_cast<long long>(k > 0 ? k : 0) * B + 127) / 128 * 128;
    return r < M ? static_cast<int>(r) : M;
}

// X of the received-workers pass: row m of slot s = m / B < k is pool row
// idx[sel[s] B + m % B] (an index outside [0, S) reads row 0); rows from k B up to
// the live row count are zero; later rows are not written.
struct ReceivedRows {
    const int32_t* idx;
    const int32_t* sel;
    const int* kdev;
    int B;
    int64_t S;
    __device__ int live(int rows) const { return live_rows(kdev, B, rows); }
    __device__ int64_t operator()(int m) const {
        const int s = m / B;
        if (s >= *kdev) return -1;
        const int64_t r = idx[static_cast<int64_t>(sel[s]) * B + (m - s * B)];
        return (r < 0 || r >= S) ? 0 : r;
    }
};

// dst [cols, ldd] = src [rows, lds]^T  (bf16), rows x cols logical; with kdev, only
// the live rows (live_rows) are transposed.
__global__ void transpose_bf16_kernel(const __nv_bfloat16* __restrict__ src, int rows, int cols, int64_t lds,
                                      __nv_bfloat16* __restrict__ dst, int64_t ldd, const int* kdev = nullptr,
                                      int B = 0) {
    __shared__ __nv_bfloat16 tile[32][33];
    const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
    rows = live_rows(kdev, B, rows);
    if (r0 >= rows) return;
    const int tx = threadIdx.x, ty = threadIdx.y;
    for (int r = ty; r < 32; r += 8) {
        const int rr = r0 + r, cc = c0 + tx;
        tile[r][tx] = (rr < rows && cc < cols) ? src[static_cast<int64_t>(rr) * lds + cc] : __float2bfloat16_rn(0.f);
    }
    __syncthreads();
    for (int r = ty; r < 32; r += 8) {
        const int cc = c0 + r, rr = r0 + tx;
        if (cc < cols && rr < rows) dst[static_cast<int64_t>(cc) * ldd + rr] = tile[tx][r];
    }
}

// With ``sel`` (received-workers pass): CTA s handles slot s, i.e. worker sel[s]
// (stacked rows s B .., samples idx[sel[s] B + r], loss[sel[s]]); slots s >= k
// zero their dZ rows up to the live row count and stop.
// With ``dZT`` the CTA also writes its rows of the transposed copy dZT [C, ldT]
// (columns i B .. i B + B - 1): the bf16 values go through a [B, C + 8] shared tile
// (dynamic shared memory) and leave as 16-byte pieces of 8 rows.
__device__ __forceinline__ void write_dzT(const __nv_bfloat16* tile, int C, int B, int64_t col0, int rows_live,
                                          __nv_bfloat16* __restrict__ dZT, int64_t ldT) {
    const int groups = B / 8;   // B % 32 == 0 on the tcgen05 path
    for (int q = threadIdx.x; q < C * groups; q += blockDim.x) {
        const int c = q / groups, g8 = q % groups;
        if (8 * g8 >= rows_live) continue;
        uint4 v;
        __nv_bfloat16* h = reinterpret_cast<__nv_bfloat16*>(&v);
#pragma unroll
        for (int t = 0; t < 8; ++t) h[t] = tile ? tile[(8 * g8 + t) * (C + 8) + c] : __float2bfloat16_rn(0.f);
        *reinterpret_cast<uint4*>(dZT + static_cast<int64_t>(c) * ldT + col0 + 8 * g8) = v;
    }
}

__global__ void __launch_bounds__(256) softmax_xent_ld_kernel(const float* __restrict__ logits, int64_t ldl, int C,
                                                              int B, const int32_t* __restrict__ idx, int64_t S,
                                                              const int32_t* __restrict__ labels,
                                                              float* __restrict__ sample_loss,
                                                              __nv_bfloat16* __restrict__ dZ, int64_t ldz,
                                                              float* __restrict__ loss,
                                                              const int32_t* __restrict__ sel = nullptr,
                                                              const int* __restrict__ kdev = nullptr,
                                                              __nv_bfloat16* __restrict__ dZT = nullptr,
                                                              int64_t ldT = 0) {
    extern __shared__ __nv_bfloat16 tileT[];   // [B][C + 8] when dZT is given
    const int i = blockIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    int worker = i;
    if (sel) {
        if (i >= *kdev) {
            const int live = live_rows(kdev, B, gridDim.x * B);
            for (int r = warp; r < B && i * B + r < live; r += nw)
                for (int c = lane; c < C; c += 32)
                    dZ[(static_cast<int64_t>(i) * B + r) * ldz + c] = __float2bfloat16_rn(0.f);
            if (dZT) write_dzT(nullptr, C, B, static_cast<int64_t>(i) * B, live - i * B, dZT, ldT);
            return;
        }
        worker = sel[i];
    }
    __shared__ int bad_s;
    constexpr int kShared = 1024;   // sample losses kept in shared memory up to this B
    __shared__ float ls[kShared];
    if (threadIdx.x == 0) bad_s = 0;
    __syncthreads();
    const float invB = 1.0f / static_cast<float>(B);
    constexpr int kRegs = 32;   // logits a lane keeps in registers: rows of up to 1024 classes in one read
    for (int r = warp; r < B; r += nw) {
        const int64_t row = static_cast<int64_t>(i) * B + r;
        const int64_t sidx = idx[static_cast<int64_t>(worker) * B + r];
        int y = -1;
        if (sidx >= 0 && sidx < S) y = labels[sidx];
        const bool bad = (y < 0 || y >= C);
        const float* z = logits + row * ldl;
        float mx = -INFINITY, se = 0.f;
        if (C <= 32 * kRegs) {
            // the row is read once: max, sum of exponentials and dZ from registers
            float v[kRegs];
#pragma unroll
            for (int j = 0; j < kRegs; ++j) {
                const int c = lane + 32 * j;
                v[j] = c < C ? z[c] : -INFINITY;
                mx = fmaxf(mx, v[j]);
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
#pragma unroll
            for (int j = 0; j < kRegs; ++j) {
                v[j] = lane + 32 * j < C ? expf(v[j] - mx) : 0.f;
                se += v[j];
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) se += __shfl_xor_sync(0xffffffffu, se, o);
            const float inv_se = 1.0f / se;
#pragma unroll
            for (int j = 0; j < kRegs; ++j) {
                const int c = lane + 32 * j;
                if (c < C) {
                    float g = v[j] * inv_se;
                    if (c == y) g -= 1.0f;
                    const __nv_bfloat16 h = __float2bfloat16_rn(bad ? NAN : g * invB);
                    dZ[row * ldz + c] = h;
                    if (dZT) tileT[r * (C + 8) + c] = h;
                }
            }
        } else {
            for (int c = lane; c < C; c += 32) mx = fmaxf(mx, z[c]);
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
            for (int c = lane; c < C; c += 32) se += expf(z[c] - mx);
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) se += __shfl_xor_sync(0xffffffffu, se, o);
            const float inv_se = 1.0f / se;
            for (int c = lane; c < C; c += 32) {
                float g = expf(z[c] - mx) * inv_se;
                if (c == y) g -= 1.0f;
                const __nv_bfloat16 h = __float2bfloat16_rn(bad ? NAN : g * invB);
                dZ[row * ldz + c] = h;
                if (dZT) tileT[r * (C + 8) + c] = h;
            }
        }
        if (lane == 0) {
            const float l = bad ? NAN : (mx + logf(se)) - z[y];
            sample_loss[row] = l;
            if (r < kShared) ls[r] = l;
            if (bad) bad_s = 1;
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        // in sample order, from shared memory
        float acc = 0.f;
        for (int r = 0; r < B; ++r) acc += r < kShared ? ls[r] : sample_loss[static_cast<int64_t>(i) * B + r];
        loss[worker] = bad_s ? NAN : acc * invB;
    }
    if (dZT) write_dzT(tileT, C, B, static_cast<int64_t>(i) * B, B, dZT, ldT);
}

// Shared memory of softmax_xent_ld_kernel's transposing tile, or 0 when it does not
// fit (the transpose then runs as transpose_bf16_kernel).
inline int softmax_tile_bytes(int B, int C) {
    const long long bytes = static_cast<long long>(B) * (C + 8) * 2;
    return bytes <= 160 * 1024 ? static_cast<int>(bytes) : 0;
}

// G[i, offb + o] = sum_{r < B} dZ[i*B + r, o] (rows in order).
__global__ void bias_grad_ld_kernel(const __nv_bfloat16* __restrict__ dZ, int64_t ldz, int out, int B,
                                    float* __restrict__ G, int64_t ldG, int64_t offb) {
    const int i = blockIdx.y;
    const int o = blockIdx.x * blockDim.x + threadIdx.x;
    if (o >= out) return;
    const __nv_bfloat16* p = dZ + static_cast<int64_t>(i) * B * ldz + o;
    float acc = 0.f;
    for (int r = 0; r < B; ++r) acc += __bfloat162float(p[static_cast<int64_t>(r) * ldz]);
    G[static_cast<int64_t>(i) * ldG + offb + o] = acc;
}

// ------------------------------------------------------------------ received-workers pass
// sel[0..k) = the workers with mask[j] != 0 in increasing order, *kout = k, and
// loss[j] = NaN for the others (their gradients are never formed).  One CTA of
// 1024 threads: a ballot prefix count per warp, then over the warp totals.
__global__ void __launch_bounds__(1024) compact_received_kernel(const uint8_t* __restrict__ mask, int n,
                                                                int32_t* __restrict__ sel, int* __restrict__ kout,
                                                                float* __restrict__ loss, int* __restrict__ zero,
                                                                int nzero) {
    __shared__ int warp_tot[32];
    const int j = threadIdx.x, lane = j & 31, warp = j >> 5;
    for (int q = j; q < nzero; q += blockDim.x) zero[q] = 0;
    const bool on = j < n && mask[j] != 0;
    const unsigned bal = __ballot_sync(0xffffffffu, on);
    if (lane == 0) warp_tot[warp] = __popc(bal);
    __syncthreads();
    int base = 0;
    for (int q = 0; q < warp; ++q) base += warp_tot[q];
    if (on) sel[base + __popc(bal & ((1u << lane) - 1u))] = j;
    else if (j < n) loss[j] = NAN;
    if (j == 0) {
        int k = 0;
        for (int q = 0; q < 32; ++q) k += warp_tot[q];
        *kout = k;
    }
}

// Bias part of Eqs. (3)-(4), g[o] = (1/k) sum_{r < k B} dZ[r, o], for every layer,
// in two launches.  The layers' blocks sit side by side in x; a block finds its
// layer in the prefix table cb0 (blocks of 256 columns).
struct BiasLayers {
    int L;
    const __nv_bfloat16* dz[DBW_LMAX];   // dZ_l [M, ldz]
    int64_t ldz;
    int out[DBW_LMAX];
    int cb0[DBW_LMAX + 1];               // first column block of layer l; cb0[L] = all blocks
    float* part[DBW_LMAX];               // [chunks, out_l] column sums per 256-row chunk
    float* wb[DBW_LMAX];                 // b_l inside w
    float* gb[DBW_LMAX];                 // b_l inside g_t (nullable)
    double* pieces[DBW_LMAX];            // [column blocks of layer l]: pieces of ||g_t(b_l)||^2
};

__device__ __forceinline__ int bias_layer(const BiasLayers& a, int blk) {
    int l = 0;
    while (l + 1 < a.L && blk >= a.cb0[l + 1]) ++l;
    return l;
}

// bias_rows_kernel: one CTA per (layer, 256 columns, 256-row chunk); thread (warp y,
// lane) sums 8 columns (16-byte loads) over rows y, y + 8, ... of the chunk, and the 8
// warps' sums are added in warp order into part[chunk][o].  Chunks past k B write
// nothing.
__global__ void __launch_bounds__(256) bias_rows_kernel(BiasLayers a, int B, const int* __restrict__ kdev) {
    __shared__ float red[8][256];
    const int k = *kdev;
    const int rows = k > 0 ? k * B : 0;
    const int r0 = blockIdx.y * 256;
    if (r0 >= rows) return;
    const int l = bias_layer(a, blockIdx.x);
    const int cb = blockIdx.x - a.cb0[l], out = a.out[l];
    const __nv_bfloat16* dZ = a.dz[l];
    const int64_t ldz = a.ldz;
    const int lane = threadIdx.x & 31, y = threadIdx.x >> 5;
    const int c = cb * 256 + 8 * lane;
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    const int rend = r0 + 256 < rows ? r0 + 256 : rows;
    if (c + 7 < out) {
#pragma unroll 4
        for (int r = r0 + y; r < rend; r += 8) {
            const uint4 raw = *reinterpret_cast<const uint4*>(dZ + static_cast<int64_t>(r) * ldz + c);
            const __nv_bfloat16* h = reinterpret_cast<const __nv_bfloat16*>(&raw);
#pragma unroll
            for (int j = 0; j < 8; ++j) acc[j] += __bfloat162float(h[j]);
        }
    } else {
        for (int r = r0 + y; r < rend; r += 8)
            for (int j = 0; j < 8 && c + j < out; ++j) acc[j] += __bfloat162float(dZ[static_cast<int64_t>(r) * ldz + c + j]);
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) red[y][8 * lane + j] = acc[j];
    __syncthreads();
    const int o = cb * 256 + threadIdx.x;
    if (o < out) {
        float t = 0.f;
        for (int q = 0; q < 8; ++q) t += red[q][threadIdx.x];
        a.part[l][static_cast<int64_t>(blockIdx.y) * out + o] = t;
    }
}

// bias_mean_update_kernel: one CTA per (layer, 256 columns): g[o] = (1/k) sum of the
// chunks' sums (chunk order), wb[o] -= lr g, gb[o] = g (nullable); the CTA's sum of g^2
// (fp64, fixed tree) into pieces[column block].
__global__ void __launch_bounds__(256) bias_mean_update_kernel(BiasLayers a, int B, const int* __restrict__ kdev,
                                                               float lr) {
    __shared__ double red[8];
    const int k = *kdev;
    const int chunks = k > 0 ? (k * B + 255) / 256 : 0;
    const int l = bias_layer(a, blockIdx.x);
    const int cb = blockIdx.x - a.cb0[l], out = a.out[l];
    const int o = cb * 256 + threadIdx.x;
    double sq = 0.0;
    if (o < out && k > 0) {
        float t = 0.f;
        for (int q = 0; q < chunks; ++q) t += a.part[l][static_cast<int64_t>(q) * out + o];
        const float g = t * (1.0f / static_cast<float>(k));
        a.wb[l][o] = fmaf(-lr, g, a.wb[l][o]);
        if (a.gb[l]) a.gb[l][o] = g;
        sq = static_cast<double>(g) * g;
    }
    for (int off = 16; off > 0; off >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, off);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = sq;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int w = 0; w < 8; ++w) t += red[w];
        a.pieces[l][cb] = t;
    }
}

struct FinishArgs {
    int L, n, B, CT;
    const double* pw[DBW_LMAX];   // tile pieces of ||g_t(W_l)||^2
    int64_t npw[DBW_LMAX];
    const double* pb[DBW_LMAX];   // CTA pieces of ||g_t(b_l)||^2
    int npb[DBW_LMAX];
    const double* pg[DBW_LMAX];   // Gram pieces, [(row group) * CT + ct]
};

// Writes the partials buffer dbw_grad_stats reads (one block per quantity):
//   vals[j] = ||g_j||^2 for received j (sum over layers and the worker's Gram pieces),
//             0 for the others;
//   vals[n + 1] = ||g_t||^2 (all W and b pieces);
//   vals[n] = sum_j ||g_j||^2 - k ||g_t||^2, the deviation sum of Eq. (10) by the
//             identity sum_j ||g_j - g_t||^2 = sum_j ||g_j||^2 - k ||g_t||^2 (fp64).
// Every sum runs in a fixed order (strided per thread, then a fixed tree).  1024
// threads: the ~12k pieces of the 4096-wide workload are ~12 loads per thread.
constexpr int kFinishThreads = 1024;

__global__ void __launch_bounds__(kFinishThreads) finish_received_kernel(FinishArgs a, const int32_t* __restrict__ sel,
                                                                         const int* __restrict__ kdev,
                                                                         double* __restrict__ partials) {
    __shared__ double red[2][kFinishThreads];
    const int t = threadIdx.x, n = a.n;
    const int k = *kdev;
    int64_t* hdr = reinterpret_cast<int64_t*>(partials);
    double* vals = partials + kPartialsHeader + (n + 2);
    if (t == 0) {
        hdr[0] = kPartialsMagic;
        hdr[1] = 1;
        hdr[2] = n;
        hdr[3] = 0;
    }
    for (int j = t; j < n; j += kFinishThreads) vals[j] = 0.0;
    double g2 = 0.0, rs = 0.0;
    for (int l = 0; l < a.L; ++l) {
        for (int64_t i = t; i < a.npw[l]; i += kFinishThreads) g2 += a.pw[l][i];
        for (int i = t; i < a.npb[l]; i += kFinishThreads) g2 += a.pb[l][i];
    }
    __syncthreads();   // zeros above land before the received rows below
    const int groups = a.B / 32;   // 32-row groups per worker
    for (int s = t; s < k; s += kFinishThreads) {
        double v = 0.0;
        for (int l = 0; l < a.L; ++l) {
            const double* pg = a.pg[l] + static_cast<int64_t>(s) * groups * a.CT;
            for (int i = 0; i < groups * a.CT; ++i) v += pg[i];
        }
        vals[sel[s]] = v;
        rs += v;
    }
    red[0][t] = g2;
    red[1][t] = rs;
    __syncthreads();
    for (int h = kFinishThreads / 2; h > 0; h >>= 1) {
        if (t < h) {
            red[0][t] += red[0][t + h];
            red[1][t] += red[1][t + h];
        }
        __syncthreads();
    }
    if (t == 0) {
        if (k > 0) {
            vals[n + 1] = red[0][0];
            vals[n] = red[1][0] - static_cast<double>(k) * red[0][0];
        } else {
            vals[n + 1] = NAN;
            vals[n] = NAN;
        }
    }
}

}  // namespace

bool tc_eligible(int prec, int B) { return prec == DBW_PREC_BF16 && B % 32 == 0; }

// bf16 W_l and W_l^T of every layer (one launch).
static void launch_weight_casts(const TcPlan& P, const float* w, char* ws, cudaStream_t st) {
    const GradsPlan& g = P.g;
    WeightCasts a{};
    a.L = g.L;
    a.t0[0] = 0;
    for (int l = 0; l < g.L; ++l) {
        const int fin = g.widths[l], fout = g.widths[l + 1];
        a.w[l] = w + g.offW[l];
        a.fin[l] = fin;
        a.fout[l] = fout;
        a.tx[l] = (fin + 63) / 64;
        a.t0[l + 1] = a.t0[l] + a.tx[l] * ((fout + 63) / 64);
        a.wb[l] = reinterpret_cast<__nv_bfloat16*>(ws + P.off_wb[l]);
        a.ldw[l] = P.ldw[l];
        // no input gradient is formed for the first layer: W_0^T is never read
        a.wt[l] = l == 0 ? nullptr : reinterpret_cast<__nv_bfloat16*>(ws + P.off_wt[l]);
        a.ldwt[l] = P.ldwt[l];
    }
    cast_transpose_weights_kernel<<<a.t0[g.L], 256, 0, st>>>(a);
}

bool make_tc_plan(int L, const int32_t* widths, int n, int B, TcPlan* P) {
    GradsPlan g;
    if (!make_grads_plan(L, widths, n, B, DBW_PREC_BF16, &g)) return false;
    P->g = g;
    const int64_t M = static_cast<int64_t>(n) * B;
    P->M8 = rup(M, 8);
    int maxw = 0;
    for (int l = 0; l <= L; ++l) maxw = widths[l] > maxw ? widths[l] : maxw;
    size_t cur = 0;
    auto take = [&](size_t bytes) {
        const size_t at = cur;
        cur += (bytes + 255) / 256 * 256;
        return at;
    };
    P->off_status = take(256);
    for (int l = 0; l < L; ++l) {
        const int fin = widths[l], fout = widths[l + 1];
        P->ldw[l] = rup(fin, 8);
        P->ldwt[l] = rup(fout, 8);
        P->off_wb[l] = take(static_cast<size_t>(fout) * P->ldw[l] * 2);
        P->off_wt[l] = take(static_cast<size_t>(fin) * P->ldwt[l] * 2);
    }
    for (int l = 0; l < L; ++l) {   // act[0] = X
        P->ldact[l] = rup(widths[l], 8);
        P->off_act[l] = take(static_cast<size_t>(M) * P->ldact[l] * 2);
        P->off_actT[l] = take(static_cast<size_t>(widths[l]) * P->M8 * 2);
    }
    P->ldlog = rup(widths[L], 4);
    P->off_logits = take(static_cast<size_t>(M) * P->ldlog * 4);
    P->off_sloss = take(static_cast<size_t>(M) * 4);
    P->ldz = rup(maxw, 8);
    P->off_dz[0] = take(static_cast<size_t>(M) * P->ldz * 2);
    P->off_dz[1] = take(static_cast<size_t>(M) * P->ldz * 2);
    P->off_dzT = take(static_cast<size_t>(maxw) * P->M8 * 2);
    P->ws_bytes = cur;
    return true;
}

int worker_grads_tc(const TcPlan& P, const float* w, const float* pool, int64_t S, const int32_t* labels,
                    const int32_t* idx, float* G, int64_t ld, float* loss, char* ws, cudaStream_t st) {
    const GradsPlan& g = P.g;
    const int L = g.L, M = g.M, B = g.B, n = g.n;
    int* status = reinterpret_cast<int*>(ws + P.off_status);
    auto bf = [&](size_t off) { return reinterpret_cast<__nv_bfloat16*>(ws + off); };
    cudaError_t e = cudaMemsetAsync(status, 0, sizeof(int), st);
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_worker_grads: %s", cudaGetErrorString(e));

    // bf16 weights and their transposes
    launch_weight_casts(P, w, ws, st);
    // X and X^T
    {
        const int in = g.widths[0];
        dim3 grid((in + 63) / 64, (M + 63) / 64);
        cast_transpose_tile_kernel<<<grid, 256, 0, st>>>(pool, in, M, in, GatherRows{idx, S}, bf(P.off_act[0]),
                                                         P.ldact[0], bf(P.off_actT[0]), P.M8);
    }
    e = cudaGetLastError();
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_worker_grads: %s", cudaGetErrorString(e));

    // forward
    float* logits = reinterpret_cast<float*>(ws + P.off_logits);
    for (int l = 0; l < L; ++l) {
        const int fin = g.widths[l], fout = g.widths[l + 1];
        TcEpi ep{};
        ep.bias = w + g.offb[l];
        int rc;
        if (l < L - 1) {
            ep.out = bf(P.off_act[l + 1]);
            ep.ldo = P.ldact[l + 1];
            ep.outT = bf(P.off_actT[l + 1]);
            ep.ldT = P.M8;
            rc = tc_gemm(TC_HIDDEN, bf(P.off_act[l]), P.ldact[l], M, fin, bf(P.off_wb[l]), P.ldw[l], fout, fin, M,
                         fout, fin, 1, 0, ep, status, st);
        } else {
            ep.outF = logits;
            ep.ldF = P.ldlog;
            rc = tc_gemm(TC_LOGITS, bf(P.off_act[l]), P.ldact[l], M, fin, bf(P.off_wb[l]), P.ldw[l], fout, fin, M,
                         fout, fin, 1, 0, ep, status, st);
        }
        if (rc) return rc;
    }
    // loss, dZ_L and its transpose
    const int C = g.widths[L];
    float* sloss = reinterpret_cast<float*>(ws + P.off_sloss);
    int cur = 0;
    if (const int tb = softmax_tile_bytes(B, C)) {
        e = cudaFuncSetAttribute(softmax_xent_ld_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, tb);
        if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_worker_grads: %s", cudaGetErrorString(e));
        softmax_xent_ld_kernel<<<n, 256, tb, st>>>(logits, P.ldlog, C, B, idx, S, labels, sloss, bf(P.off_dz[0]),
                                                   P.ldz, loss, nullptr, nullptr, bf(P.off_dzT), P.M8);
    } else {
        softmax_xent_ld_kernel<<<n, 256, 0, st>>>(logits, P.ldlog, C, B, idx, S, labels, sloss, bf(P.off_dz[0]),
                                                  P.ldz, loss);
        dim3 tg((C + 31) / 32, (M + 31) / 32);
        transpose_bf16_kernel<<<tg, dim3(32, 8), 0, st>>>(bf(P.off_dz[0]), M, C, P.ldz, bf(P.off_dzT), P.M8);
    }
    e = cudaGetLastError();
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_worker_grads: %s", cudaGetErrorString(e));

    // backward
    for (int l = L - 1; l >= 0; --l) {
        const int fin = g.widths[l], fout = g.widths[l + 1];
        TcEpi ep{};
        ep.G = G;
        ep.ldG = ld;
        ep.off = g.offW[l];
        ep.ldrow = fin;
        int rc = tc_gemm(TC_DW, bf(P.off_dzT), P.M8, fout, M, bf(P.off_actT[l]), P.M8, fin, M, fout, fin, B, n, B,
                         ep, status, st);
        if (rc) return rc;
        bias_grad_ld_kernel<<<dim3((fout + 127) / 128, n), 128, 0, st>>>(bf(P.off_dz[cur]), P.ldz, fout, B, G, ld,
                                                                          g.offb[l]);
        e = cudaGetLastError();
        if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_worker_grads: %s", cudaGetErrorString(e));
        if (l > 0) {
            TcEpi ex{};
            ex.act = bf(P.off_act[l]);
            ex.ldact = P.ldact[l];
            ex.out = bf(P.off_dz[cur ^ 1]);
            ex.ldo = P.ldz;
            ex.outT = bf(P.off_dzT);
            ex.ldT = P.M8;
            rc = tc_gemm(TC_DX, bf(P.off_dz[cur]), P.ldz, M, fout, bf(P.off_wt[l]), P.ldwt[l], fin, fout, M, fin,
                         fout, 1, 0, ex, status, st);
            if (rc) return rc;
            cur ^= 1;
        }
    }
    return DBW_OK;
}

// ------------------------------------------------------------------ received-workers pass
// Eqs. (2)-(4) and the statistics of Sect. 3.1 for the k received workers only,
// without the [n, d] gradient matrix: the rows of the received workers are
// stacked (slot s = s-th received worker), the forward and input-gradient GEMMs
// run over those k B rows, the weight part of g_t is one GEMM with K = k B whose
// epilogue applies the SGD step (TC_GBAR), the bias part is a column sum, and the
// per-worker squared norms come from B x B Gram matrices (tc_gram).  The number
// of received workers k is read on the device from ``mask``.

bool rx_eligible(int prec, int B) { return tc_eligible(prec, B) && (128 % B == 0 || B % 128 == 0); }

bool make_rx_plan(int L, const int32_t* widths, int n, int B, RxPlan* P) {
    if (!make_tc_plan(L, widths, n, B, &P->t)) return false;
    const GradsPlan& g = P->t.g;
    P->CT = B > 128 ? B / 128 : 1;
    size_t cur = P->t.ws_bytes;
    auto take = [&](size_t bytes) {
        const size_t at = cur;
        cur += (bytes + 255) / 256 * 256;
        return at;
    };
    P->off_sel = take(static_cast<size_t>(n) * 4);
    P->off_k = take(4);
    int maxout = 0;
    for (int l = 0; l < L; ++l) maxout = g.widths[l + 1] > maxout ? g.widths[l + 1] : maxout;
    for (int l = 0; l < L; ++l)   // bias column sums per 256-row chunk, per layer
        P->off_bpart[l] = take(static_cast<size_t>((g.M + 255) / 256) * g.widths[l + 1] * 4);
    // dZ_l of every layer stays until the bias sums and the Gram norms of all layers run
    // after the backward pass: the two ping-pong buffers hold the last two layers'
    for (int l = 0; l < L; ++l) {
        const int back = L - 1 - l;
        P->off_dzl[l] = back < 2 ? P->t.off_dz[back] : take(static_cast<size_t>(g.M) * P->t.ldz * 2);
    }
    for (int l = 0; l < L; ++l) {
        const int fin = g.widths[l], fout = g.widths[l + 1];
        P->npw[l] = static_cast<int64_t>((fout + 127) / 128) * ((fin + 255) / 256) * 8;
        P->off_pw[l] = take(static_cast<size_t>(P->npw[l]) * 8);
        P->npb[l] = (fout + 255) / 256;
        P->off_pb[l] = take(static_cast<size_t>(P->npb[l]) * 8);
        P->off_pg[l] = take(static_cast<size_t>(g.M / 32) * P->CT * 8);
    }
    P->off_dzT2 = take(static_cast<size_t>(maxout > g.widths[0] ? maxout : g.widths[0]) * P->t.M8 * 2);
    P->off_gpart = take(tc_gram_partial_floats(g.M, B, L) * 4);
    P->ngcnt = static_cast<int>(tc_gram_items(g.M, B, L));
    P->off_gcnt = take(static_cast<size_t>(P->ngcnt) * 4);
    P->ws_bytes = cur;
    return true;
}

int received_grads_tc(const RxPlan& P, float* w, const float* pool, int64_t S, const int32_t* labels,
                      const int32_t* idx, const uint8_t* mask, float lr, float* gbar, float* loss, double* partials,
                      char* ws, cudaStream_t st) {
    const TcPlan& T = P.t;
    const GradsPlan& g = T.g;
    const int L = g.L, M = g.M, B = g.B, n = g.n;
    int* status = reinterpret_cast<int*>(ws + T.off_status);
    int32_t* sel = reinterpret_cast<int32_t*>(ws + P.off_sel);
    int* kdev = reinterpret_cast<int*>(ws + P.off_k);
    auto bf = [&](size_t off) { return reinterpret_cast<__nv_bfloat16*>(ws + off); };
    auto f64 = [&](size_t off) { return reinterpret_cast<double*>(ws + off); };
    const char* what = "dbw_received_grads_update";
    cudaError_t e = cudaMemsetAsync(status, 0, sizeof(int), st);
    if (e != cudaSuccess) return fail(DBW_ECUDA, "%s: %s", what, cudaGetErrorString(e));

    int* gcnt = reinterpret_cast<int*>(ws + P.off_gcnt);
    float* gpart = reinterpret_cast<float*>(ws + P.off_gpart);
    compact_received_kernel<<<1, 1024, 0, st>>>(mask, n, sel, kdev, loss, gcnt, P.ngcnt);
    launch_weight_casts(T, w, ws, st);
    {
        const int in = g.widths[0];
        dim3 grid((in + 63) / 64, (M + 63) / 64);
        cast_transpose_tile_kernel<<<grid, 256, 0, st>>>(pool, in, M, in, ReceivedRows{idx, sel, kdev, B, S},
                                                         bf(T.off_act[0]), T.ldact[0], bf(T.off_actT[0]), T.M8);
    }
    e = cudaGetLastError();
    if (e != cudaSuccess) return fail(DBW_ECUDA, "%s: %s", what, cudaGetErrorString(e));

    // forward over the live rows
    float* logits = reinterpret_cast<float*>(ws + T.off_logits);
    for (int l = 0; l < L; ++l) {
        const int fin = g.widths[l], fout = g.widths[l + 1];
        TcEpi ep{};
        ep.bias = w + g.offb[l];
        ep.kdev = kdev;
        ep.kmul = B;
        int rc;
        if (l < L - 1) {
            ep.out = bf(T.off_act[l + 1]);
            ep.ldo = T.ldact[l + 1];
            ep.outT = bf(T.off_actT[l + 1]);
            ep.ldT = T.M8;
            rc = tc_gemm(TC_HIDDEN, bf(T.off_act[l]), T.ldact[l], M, fin, bf(T.off_wb[l]), T.ldw[l], fout, fin, M,
                         fout, fin, 1, 0, ep, status, st);
        } else {
            ep.outF = logits;
            ep.ldF = T.ldlog;
            rc = tc_gemm(TC_LOGITS, bf(T.off_act[l]), T.ldact[l], M, fin, bf(T.off_wb[l]), T.ldw[l], fout, fin, M,
                         fout, fin, 1, 0, ep, status, st);
        }
        if (rc) return rc;
    }
    const int C = g.widths[L];
    float* sloss = reinterpret_cast<float*>(ws + T.off_sloss);
    if (const int tb = softmax_tile_bytes(B, C)) {
        e = cudaFuncSetAttribute(softmax_xent_ld_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, tb);
        if (e != cudaSuccess) return fail(DBW_ECUDA, "%s: %s", what, cudaGetErrorString(e));
        softmax_xent_ld_kernel<<<n, 256, tb, st>>>(logits, T.ldlog, C, B, idx, S, labels, sloss,
                                                   bf(P.off_dzl[L - 1]), T.ldz, loss, sel, kdev, bf(T.off_dzT), T.M8);
    } else {
        softmax_xent_ld_kernel<<<n, 256, 0, st>>>(logits, T.ldlog, C, B, idx, S, labels, sloss, bf(P.off_dzl[L - 1]),
                                                  T.ldz, loss, sel, kdev);
        dim3 tg((C + 31) / 32, (M + 31) / 32);
        transpose_bf16_kernel<<<tg, dim3(32, 8), 0, st>>>(bf(P.off_dzl[L - 1]), M, C, T.ldz, bf(T.off_dzT), T.M8, kdev,
                                                          B);
    }
    e = cudaGetLastError();
    if (e != cudaSuccess) return fail(DBW_ECUDA, "%s: %s", what, cudaGetErrorString(e));

    // backward: per layer the mean gradient with the SGD step and dZ of the layer below in
    // one launch.  dZ_l^T alternates between two buffers: the dX GEMM writes dZ_{l-1}^T
    // into one while the mean-gradient GEMM reads dZ_l^T from the other.  dZ_l itself
    // (row-major) is kept for every layer.
    __nv_bfloat16* dzT[2] = {bf(T.off_dzT), bf(P.off_dzT2)};
    int curT = 0;
    for (int l = L - 1; l >= 0; --l) {
        const int fin = g.widths[l], fout = g.widths[l + 1];
        TcEpi gb{};
        gb.W = w;
        gb.gbar = gbar;
        gb.lr = lr;
        gb.off = g.offW[l];
        gb.ldrow = fin;
        gb.pieces = f64(P.off_pw[l]);
        gb.kdev = kdev;
        gb.kmul = B;
        const TcOperands go{dzT[curT], T.M8, fout, M, bf(T.off_actT[l]), T.M8, fin, M, fout, fin, M};
        int rc;
        if (l > 0) {
            TcEpi ex{};
            ex.act = bf(T.off_act[l]);
            ex.ldact = T.ldact[l];
            ex.out = bf(P.off_dzl[l - 1]);
            ex.ldo = T.ldz;
            ex.outT = dzT[curT ^ 1];
            ex.ldT = T.M8;
            ex.kdev = kdev;
            ex.kmul = B;
            const TcOperands xo{bf(P.off_dzl[l]), T.ldz, M, fout, bf(T.off_wt[l]), T.ldwt[l], fin, fout, M, fin, fout};
            rc = tc_gemm_mean_dx(go, gb, xo, ex, status, st);
        } else {
            rc = tc_gemm(TC_GBAR, go.A, go.lda, go.rowsA, go.colsA, go.B, go.ldb, go.rowsB, go.colsB, go.M, go.N, go.K,
                         1, 0, gb, status, st);
        }
        if (rc) return rc;
        curT ^= 1;
    }
    // bias part of g_t and its step, every layer in two launches
    {
        BiasLayers bl{};
        bl.L = L;
        bl.ldz = T.ldz;
        bl.cb0[0] = 0;
        for (int l = 0; l < L; ++l) {
            bl.dz[l] = bf(P.off_dzl[l]);
            bl.out[l] = g.widths[l + 1];
            bl.cb0[l + 1] = bl.cb0[l] + P.npb[l];
            bl.part[l] = reinterpret_cast<float*>(ws + P.off_bpart[l]);
            bl.wb[l] = w + g.offb[l];
            bl.gb[l] = gbar ? gbar + g.offb[l] : nullptr;
            bl.pieces[l] = f64(P.off_pb[l]);
        }
        bias_rows_kernel<<<dim3(bl.cb0[L], (M + 255) / 256), 256, 0, st>>>(bl, B, kdev);
        bias_mean_update_kernel<<<bl.cb0[L], 256, 0, st>>>(bl, B, kdev, lr);
        e = cudaGetLastError();
        if (e != cudaSuccess) return fail(DBW_ECUDA, "%s: %s", what, cudaGetErrorString(e));
    }
    // per-worker norms of every layer in one launch
    {
        const __nv_bfloat16* acts[DBW_LMAX];
        const __nv_bfloat16* dzs[DBW_LMAX];
        int64_t lds[DBW_LMAX];
        int cin[DBW_LMAX], cout[DBW_LMAX];
        double* pg[DBW_LMAX];
        for (int l = 0; l < L; ++l) {
            acts[l] = bf(T.off_act[l]);
            lds[l] = T.ldact[l];
            cin[l] = g.widths[l];
            dzs[l] = bf(P.off_dzl[l]);
            cout[l] = g.widths[l + 1];
            pg[l] = f64(P.off_pg[l]);
        }
        const int rc = tc_gram(L, acts, lds, cin, dzs, T.ldz, cout, M, B, kdev, pg, gpart, gcnt, status, st);
        if (rc) return rc;
    }
    FinishArgs fa{};
    fa.L = L;
    fa.n = n;
    fa.B = B;
    fa.CT = P.CT;
    for (int l = 0; l < L; ++l) {
        fa.pw[l] = f64(P.off_pw[l]);
        fa.npw[l] = P.npw[l];
        fa.pb[l] = f64(P.off_pb[l]);
        fa.npb[l] = P.npb[l];
        fa.pg[l] = f64(P.off_pg[l]);
    }
    finish_received_kernel<<<1, kFinishThreads, 0, st>>>(fa, sel, kdev, partials);
    e = cudaGetLastError();
    if (e != cudaSuccess) return fail(DBW_ECUDA, "%s: %s", what, cudaGetErrorString(e));
    return DBW_OK;
}

size_t received_workspace_bytes(int L, const int32_t* widths, int n, int B, int prec) {
    RxPlan P;
    if (!rx_eligible(prec, B) || !make_rx_plan(L, widths, n, B, &P)) return 0;
    return P.ws_bytes;
}

int launch_received_grads(int L, const int32_t* widths, int prec, float* w, int64_t d, const float* pool, int64_t S,
                          const int32_t* labels, const int32_t* idx, int n, int B, const uint8_t* mask, float lr,
                          float* gbar, float* loss, double* partials, void* ws, size_t ws_bytes, cudaStream_t st) {
    const char* what = "dbw_received_grads_update";
    if (!rx_eligible(prec, B))
        return fail(DBW_EUNSUPPORTED, "%s: needs prec = DBW_PREC_BF16, B %% 32 == 0 and B | 128 or 128 | B", what);
    RxPlan P;
    if (!make_rx_plan(L, widths, n, B, &P)) return fail(DBW_EINVAL, "%s: invalid model shape", what);
    if (d != P.t.g.d) return fail(DBW_EINVAL, "%s: d = %lld, the widths give %lld", what, (long long)d,
                                  (long long)P.t.g.d);
    if (ws_bytes < P.ws_bytes) return fail(DBW_EINVAL, "%s: workspace %zu bytes < %zu needed", what, ws_bytes, P.ws_bytes);
    return received_grads_tc(P, w, pool, S, labels, idx, mask, lr, gbar, loss, partials, static_cast<char*>(ws), st);
}

}  // namespace dbw
