// Internal plan of the worker-gradient pass: layer offsets and workspace layout.
#pragma once

#include <stddef.h>
#include <stdint.h>

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
    size_t ws_bytes;
};

bool make_grads_plan(int L, const int32_t* widths, int n, int B, int prec, GradsPlan* P);

}  // namespace dbw
