// Internal plan of the worker-gradient pass: layer offsets and workspace layout.
#pragma once

#include <stddef.h>
#include <stdint.h>

#include <cuda_runtime.h>

#include "dbw.h"

namespace dbw {

struct GradsPlan {
    int L, n, B, M, prec;
    int widths[DBW_LMAX + 1];
    int64_t offW[DBW_LMAX], offb[DBW_LMAX];   // offsets of W_l and b_l in w / in a row of G
    int64_t d;
    // workspace byte offsets (256-byte aligned)
    size_t off_x;                   // X = gathered inputs [M, widths[0]] (operand type)
    size_t off_act[DBW_LMAX];       // A_l [M, widths[l]] for l = 1..L-1 (off_act[0] = off_x)
    size_t off_logits;              // [M, C] fp32
    size_t off_sloss;               // [M] fp32 per-sample loss
    size_t off_dz[2];               // ping-pong dZ [M, max width] (operand type)
    size_t off_wb;                  // bf16 weights [d] (bf16 only)
    size_t off_split;               // split-K partial tiles of the SIMT GEMMs
    size_t split_floats;
    // fp32 forward GEMMs on the tensor cores in three tf32 passes (gemm_tf32.cuh):
    // tf32[l] says layer l's forward GEMM takes that path; its operands' hi / lo parts
    // go to off_ahi / off_alo ([M, ceil4(in)]) and off_whi / off_wlo ([out, ceil4(in)])
    bool tf32[DBW_LMAX];
    size_t off_ahi, off_alo, off_whi, off_wlo;
    // per-worker weight gradients in three tf32 passes: tf32_dw[l]; the transposed hi / lo
    // parts of dZ_l ([out, M]) and of the layer input ([in, M])
    bool tf32_dw[DBW_LMAX];
    size_t off_zthi, off_ztlo, off_athi, off_atlo;
    size_t off_xthi, off_xtlo;      // the first layer's input parts [in, M], written by the gather
    size_t ws_bytes;
};

bool make_grads_plan(int L, const int32_t* widths, int n, int B, int prec, GradsPlan* P);

// Workspace of the tcgen05 (bf16) pass; every offset 256-byte aligned, every
// leading dimension (ld*) a multiple of 8 elements.
struct TcPlan {
    GradsPlan g;                       // shapes and parameter offsets
    int64_t M8;                        // leading dimension of the transposed [width, M] buffers
    size_t off_status;                 // device int: bit 0 = a pipeline wait timed out
    size_t off_wb[DBW_LMAX];           // W_l bf16 [out, ldw]
    int64_t ldw[DBW_LMAX];
    size_t off_wt[DBW_LMAX];           // W_l^T bf16 [in, ldwt]
    int64_t ldwt[DBW_LMAX];
    size_t off_act[DBW_LMAX];          // layer-l input bf16 [M, ldact] (act[0] = X)
    int64_t ldact[DBW_LMAX];
    size_t off_actT[DBW_LMAX];         // its transpose bf16 [width, M8]
    size_t off_logits;                 // fp32 [M, ldlog]
    int64_t ldlog;
    size_t off_sloss;                  // fp32 [M]
    size_t off_dz[2];                  // bf16 [M, ldz] ping-pong
    int64_t ldz;
    size_t off_dzT;                    // bf16 [max width, M8]
    size_t ws_bytes;
};

// Workspace of the received-workers pass (dbw_received_grads_update): the bf16
// plan above (its buffers hold the k received workers' rows, slot s = the s-th
// received worker in increasing index order, at rows s B .. s B + B - 1), then:
struct RxPlan {
    TcPlan t;
    int CT;                            // Gram column tiles per 128-row tile: max(1, B / 128)
    size_t off_sel;                    // int32 [n]: received workers, increasing
    size_t off_k;                      // int32: k
    size_t off_bpart[DBW_LMAX];        // fp32 [ceil(M / 256), out_l]: bias column sums per 256-row chunk
    size_t off_dzl[DBW_LMAX];          // bf16 [M, ldz]: dZ_l of every layer (the last two in off_dz)
    size_t off_pw[DBW_LMAX];           // fp64 [tiles_l * 8]: pieces of ||g_t(W_l)||^2
    int64_t npw[DBW_LMAX];
    size_t off_pb[DBW_LMAX];           // fp64 [ceil(out_l / 256)]: pieces of ||g_t(b_l)||^2
    int npb[DBW_LMAX];
    size_t off_pg[DBW_LMAX];           // fp64 [(M / 32) * CT]: Gram pieces of ||g_j||^2
    size_t off_dzT2;                   // bf16 [max width, M8]: second dZ^T buffer (the dX GEMM of a layer
                                       // writes dZ_{l-1}^T while the mean-gradient GEMM reads dZ_l^T)
    size_t off_gpart;                  // fp32: partial Gram products of the K ranges (shared by the layers)
    size_t off_gcnt;                   // int32 [gram items]: per-item range counters, zeroed at the start of a call
    int ngcnt;
    size_t ws_bytes;
};

// The received-workers pass needs the tcgen05 path and a Gram tile layout: B % 32 == 0
// and either 128 % B == 0 or B % 128 == 0.
bool rx_eligible(int prec, int B);
bool make_rx_plan(int L, const int32_t* widths, int n, int B, RxPlan* P);
int received_grads_tc(const RxPlan& P, float* w, const float* pool, int64_t S, const int32_t* labels,
                      const int32_t* idx, const uint8_t* mask, float lr, float* gbar, float* loss, double* partials,
                      char* ws, cudaStream_t st);

// The bf16 pass runs on tcgen05 when each worker's sample count is whole 32-deep K blocks.
bool tc_eligible(int prec, int B);
bool make_tc_plan(int L, const int32_t* widths, int n, int B, TcPlan* P);
int worker_grads_tc(const TcPlan& P, const float* w, const float* pool, int64_t S, const int32_t* labels,
                    const int32_t* idx, float* G, int64_t ld, float* loss, char* ws, cudaStream_t st);

}  // namespace dbw
